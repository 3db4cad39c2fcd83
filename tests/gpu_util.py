"""Helpers of the GPU tests: seeded inputs on the device, calls through the C
ABI, comparisons with the fp64 oracle."""
from __future__ import annotations

import numpy as np
import torch

from paper_2606_19528_gb300 import lora, synth

# Tolerances of the parity bar: relative Frobenius error against the fp64
# oracle, <= 5e-3 for the bf16 outputs y, su and dx and <= 1e-2 for the fp32
# gradients dA and dB.  Expected errors are ~1e-3: bf16 rounds each output
# once (unit roundoff 2^-9; RMS relative error ~1.1e-3 for a uniform
# mantissa), and dA / dB inherit the bf16 rounding of su and sv.
TOL_Y = 5e-3
TOL_DX = 5e-3
TOL_SU = 5e-3
TOL_GRAD = 1e-2


def dev_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to("cuda").view(torch.bfloat16)


def host_f64(t: torch.Tensor) -> np.ndarray:
    if t.dtype == torch.bfloat16:
        return synth.bf16_bits_to_f64(t.view(torch.int16).cpu().numpy().view(np.uint16))
    return t.double().cpu().numpy()


def rel_fro(got, want) -> float:
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    d = np.linalg.norm(want)
    if d == 0.0:
        return float(np.linalg.norm(got))
    return float(np.linalg.norm(got - want) / d)


class DevProj:
    """Device buffers of one projection: inputs from bf16 bits, outputs allocated."""

    def __init__(self, x, W, A, B, dy, s, share_x: torch.Tensor | None = None):
        self.bits = {"x": x, "W": W, "A": A, "B": B, "dy": dy}
        self.T, self.K = x.shape
        self.N = W.shape[0]
        self.r = A.shape[0]
        self.s = float(s)
        self.x = share_x if share_x is not None else dev_bf16(x)
        self.W, self.A, self.B, self.dy = dev_bf16(W), dev_bf16(A), dev_bf16(B), dev_bf16(dy)
        dev = "cuda"
        # NaN canaries: every output element must be written
        self.y = torch.full((self.T, self.N), float("nan"), dtype=torch.bfloat16, device=dev)
        self.su = torch.full((self.T, self.r), float("nan"), dtype=torch.bfloat16, device=dev)
        self.dx = torch.full((self.T, self.K), float("nan"), dtype=torch.bfloat16, device=dev)
        self.dA = torch.full((self.r, self.K), float("nan"), dtype=torch.float32, device=dev)
        self.dB = torch.full((self.N, self.r), float("nan"), dtype=torch.float32, device=dev)

    @property
    def shape(self):
        return lora.make_shape(self.T, self.K, self.N, self.r, self.s)

    def proj(self, with_dx=True):
        return lora.make_proj(self.shape, x=self.x, W=self.W, A=self.A, B=self.B, dy=self.dy, y=self.y, su=self.su,
                              dx=self.dx if with_dx else None, dA=self.dA, dB=self.dB)

    def f64(self, name):
        return synth.bf16_bits_to_f64(self.bits[name])


def workspace(nbytes: int) -> torch.Tensor:
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device="cuda")


def run_single(p: DevProj, fwd=True, bwd=True, with_dx=True):
    st = p.shape
    if fwd:
        n = lora.lora_workspace_size(st, lora.LORA_FWD)
        ws = workspace(n)
        lora.lora_linear_fwd(st, p.x, p.W, p.A, p.B, p.y, p.su, ws, ws.numel())
    if bwd:
        n = lora.lora_workspace_size(st, lora.LORA_BWD)
        ws = workspace(n)
        lora.lora_linear_bwd(st, p.dy, p.x, p.W, p.A, p.B, p.su, p.dx if with_dx else None, p.dA, p.dB, ws,
                             ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK


def run_stack(ps, mode=lora.LORA_FWD_BWD):
    projs = [p.proj() for p in ps]
    n = lora.lora_stack_workspace_size(projs, mode)
    ws = workspace(n)
    lora.lora_stack_step(projs, mode, ws, ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK


def sample_rows(T: int, n: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    rows = set([0, T - 1, min(T - 1, 127), min(T - 1, 128)])
    rows.update(int(v) for v in rng.integers(0, T, n))
    return np.array(sorted(rows))
