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

Algorithm 1 ("On-the-fly Dequantization") stores the frozen W as integer
codes W_q with quantization parameters s, b and uses W = s W_q + b for both
the forward and the backward; `dequant_q4` is that definition for the 4-bit
layout of the CUDA library's interface (codes 0..15, one (s, b) pair per
output row and group of 64 input columns; the paper fixes neither).

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


def unpack_q4(codes) -> np.ndarray:
    """Codes [N, K] (integers 0..15) from the packed bytes [N, K / 2].

    Layout: the little-endian 32-bit word m of a row holds the codes of
    columns 8m .. 8m + 7; column 8m + 2i sits in bits 4i .. 4i + 3 and column
    8m + 2i + 1 in bits 16 + 4i .. 16 + 4i + 3 (i = 0..3)."""
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    N, half = c.shape
    words = c.view("<u4").astype(np.int64)  # [N, K / 8]
    q = np.empty((N, words.shape[1], 8), dtype=np.int64)
    for i in range(4):
        q[:, :, 2 * i] = (words >> (4 * i)) & 15
        q[:, :, 2 * i + 1] = (words >> (16 + 4 * i)) & 15
    return q.reshape(N, 2 * half)


def dequant_q4(codes, s, b) -> np.ndarray:
    """Algorithm 1's dequantization W = s * W_q + b in fp64.

    codes: packed bytes [N, K / 2] (see unpack_q4); s, b: [N, K / 64] per
    output row and group of 64 consecutive input columns."""
    q = unpack_q4(codes).astype(np.float64)
    s, b = _f64(s), _f64(b)
    g = np.arange(q.shape[1]) // 64
    return s[:, g] * q + b[:, g]
