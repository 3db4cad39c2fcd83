"""GPU test of lora_linear_fwd_noalloc: the forward for callers that cannot
allocate device memory when they call it (an operator inside another
framework's execution callback, a latency-bound path that cannot afford the
synchronisation of cudaMalloc).  Its scratch is a fixed array inside the
library instead of a caller workspace.  Its output must match the ordinary
forward (which takes a workspace) within the parity tolerances, on two calls
in a row, since every call reuses the array the previous one left behind.
This file is collected last on purpose: it runs after every other test in a
full run, and also passes alone in a fresh process."""
import numpy as np
import pytest
import torch

from paper_2606_19528_gb300 import lora, synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

CASES = [
    (512, 3072, 3072, 16),   # a q projection of the Llama-shaped layer
    (136, 200, 264, 24),     # tails in every tile dimension
    (264, 72, 520, 4),       # rank that is not a multiple of 8 (padded copies in the scratch)
]


def _inputs(T, K, N, r, seed):
    x = synth.gen_x(seed, 11, 0, 0, T, K)
    W = synth.gen_W(seed, 11, 0, 0, N, K)
    A = synth.gen_A(seed, 11, 0, 0, r, K)
    B = synth.gen_B(seed, 11, 0, 0, N, r)
    dy = synth.gen_dy(seed, 11, 0, 0, T, N)
    return x, W, A, B, dy


@pytest.mark.parametrize("T,K,N,r", CASES, ids=[f"T{t}_K{k}_N{n}_r{r}" for t, k, n, r in CASES])
def test_noalloc_forward_matches_workspace_forward(T, K, N, r):
    s = 2.0
    p = G.DevProj(*_inputs(T, K, N, r, seed=T + r), s)
    st = p.shape
    ws = G.workspace(lora.lora_workspace_size(st, lora.LORA_FWD))
    lora.lora_linear_fwd(st, p.x, p.W, p.A, p.B, p.y, p.su, ws, ws.numel())
    torch.cuda.synchronize()
    y_ref, su_ref = G.host_f64(p.y), G.host_f64(p.su)
    for call in range(2):
        y = torch.full_like(p.y, float("nan"))
        su = torch.full_like(p.su, float("nan"))
        lora.lora_linear_fwd_noalloc(st, p.x, p.W, p.A, p.B, y, su)
        torch.cuda.synchronize()
        assert lora.lora_read_status() == lora.LORA_OK
        assert not torch.isnan(y).any() and not torch.isnan(su).any(), call
        assert G.rel_fro(G.host_f64(y), y_ref) <= G.TOL_Y, call
        assert G.rel_fro(G.host_f64(su), su_ref) <= G.TOL_SU, call


def test_noalloc_rejects_shapes_beyond_its_scratch():
    # 16384 tokens x d_in 8192 at rank 64 needs far more than the fixed array
    T, K, N, r = 16384, 8192, 64, 64
    st = lora.make_shape(T, K, N, r, 2.0)
    small = torch.zeros(256, dtype=torch.bfloat16, device="cuda")
    y = torch.full((256,), float("nan"), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd_noalloc(st, small, small, small, small, y, None)
    assert e.value.code == lora.LORA_ESCRATCH
    torch.cuda.synchronize()
    assert torch.isnan(y).all(), "a rejected call must enqueue nothing"
