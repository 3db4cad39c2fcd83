"""fp64 CPU oracle of the LoRA-adapted linear layer (forward and backward).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports, links or
runs this module: only the tests, the smoke check and the benchmark's CPU
baseline arm use it.  It shares no code with the CUDA library.

What it computes.  The fine-tuning method adapts frozen linear layers with
LoRA (Background, "Parameter-Efficient Fine-Tuning": low-rank decomposition
matrices trained while the original weights stay frozen; rank r and alpha
from the hyper-parameter table).  The paper does not write the LoRA
equations out; the oracle uses the standard definition of the cited LoRA
method, in the row-major token-major layout (x is [T, d_in]; W is
[d_out, d_in] as in nn.Linear; A is [r, d_in]; B is [d_out, r]; s = alpha/r):

    u  = x A^T                  y  = x W^T + s u B^T
    v  = dy B                   dx = dy W + s v A
    dB = s dy^T u               dA = s v^T x

y = x W^T and dx = dy W are Algorithm 1's y_base = W x and dx = W^T dy
(column-vector form) transposed to this layout.  W is frozen, so dW is never
formed (Section "Base Model Quantization": the base weights stay frozen).

Every function below is the plain definition: fp64 arithmetic on inputs that
are exactly widened from bf16, with numpy's matrix product as the only
library step; no blocking, fusion or reordering.  Pins that hold it to
something other than itself (brute-force loops, a hand-worked example,
finite differences, the merged-weight identity, the full-gradient
factorisation, the B = 0 initialisation invariant) live in the test suite.
"""
from __future__ import annotations

import numpy as np


def _f64(a) -> np.ndarray:
    return np.asarray(a, dtype=np.float64)


def lora_forward(x, W, A, B, s: float):
    """Forward of the LoRA linear: returns (y, u) with u = x A^T, y = x W^T + s u B^T."""
    x, W, A, B = _f64(x), _f64(W), _f64(A), _f64(B)
    u = x @ A.T
    y = x @ W.T + s * (u @ B.T)
    return y, u


def lora_backward(dy, x, W, A, B, s: float):
    """Backward of the LoRA linear with W frozen: returns (dx, dA, dB, v).

    v = dy B; dx = dy W + s v A; dB = s dy^T (x A^T); dA = s v^T x."""
    dy, x, W, A, B = _f64(dy), _f64(x), _f64(W), _f64(A), _f64(B)
    u = x @ A.T
    v = dy @ B
    dx = dy @ W + s * (v @ A)
    dB = s * (dy.T @ u)
    dA = s * (v.T @ x)
    return dx, dA, dB, v


def lora_forward_rows(rows, x, W, A, B, s: float):
    """Rows `rows` of y only (each output row depends on its own token only)."""
    xr = _f64(x)[rows]
    A, B, W = _f64(A), _f64(B), _f64(W)
    return xr @ W.T + s * ((xr @ A.T) @ B.T)


def lora_backward_dx_rows(rows, dy, W, A, B, s: float):
    """Rows `rows` of dx only."""
    dyr = _f64(dy)[rows]
    A, B, W = _f64(A), _f64(B), _f64(W)
    return dyr @ W + s * ((dyr @ B) @ A)


def lora_adapter_grads(dy, x, A, B, s: float):
    """dA and dB alone (no dx): the reductions over tokens, O(T r (d_in + d_out))."""
    dy, x, A, B = _f64(dy), _f64(x), _f64(A), _f64(B)
    u = x @ A.T
    v = dy @ B
    return s * (v.T @ x), s * (dy.T @ u)


def lora_step(proj_inputs, s: float):
    """Forward then backward of several independent projections (a decoder
    layer's adapted linears); returns a list of dicts y, u, dx, dA, dB."""
    out = []
    for p in proj_inputs:
        y, u = lora_forward(p["x"], p["W"], p["A"], p["B"], s)
        dx, dA, dB, _ = lora_backward(p["dy"], p["x"], p["W"], p["A"], p["B"], s)
        out.append({"y": y, "u": u, "dx": dx, "dA": dA, "dB": dB})
    return out
