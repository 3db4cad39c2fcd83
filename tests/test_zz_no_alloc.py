"""GPU test of lora_linear_fwd_noalloc: the forward for callers that cannot
allocate device memory when they call it (an operator inside another
framework's execution callback, where allocating is not allowed, or a
latency-bound path that cannot afford the synchronisation cudaMalloc and
cudaFree cause).  Its scratch is a fixed array inside the library instead of
a caller workspace.  Every call reuses the array the previous call left
behind, so each case runs two calls in a row.

What must hold: with 76 or more output tiles the ordinary forward never
splits its contraction, and the two forwards run the same kernels on the same
plan, so y and su are equal bit for bit; with fewer tiles the ordinary
forward may split the contraction into fp32 partial sums while this one
never does, so they agree within the parity tolerances.  Every case is also
checked against the fp64 oracle.

This file is collected last on purpose: it runs after every other test in a
full run, and also passes alone in a fresh process."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_19528_gb300 import lora, synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

TILES = (256, 512)  # output tile of the fused contraction
PAIRS = 76          # CTA pairs of a GB300: at least this many tiles never split

CASES = [
    # T, K, N, r
    (2048, 1024, 5120, 16),   # 8 x 10 = 80 tiles: never split
    (2056, 200, 9736, 24),    # 9 x 20 tiles with tails in every dimension
    (2048, 72, 10240, 4),     # rank not a multiple of 8 (padded copies in the scratch)
    (512, 3072, 3072, 16),    # a q projection of the Llama-shaped layer: 12 tiles, may split
    (136, 200, 264, 24),      # one tile
]


def _tiles(T, N):
    return -(-T // TILES[0]) * -(-N // TILES[1])


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
    bitwise = _tiles(T, N) >= PAIRS
    y_want, u = oracle.lora_forward(p.f64("x"), p.f64("W"), p.f64("A"), p.f64("B"), s)
    for call in range(2):
        y = torch.full_like(p.y, float("nan"))
        su = torch.full_like(p.su, float("nan"))
        lora.lora_linear_fwd_noalloc(st, p.x, p.W, p.A, p.B, y, su)
        torch.cuda.synchronize()
        assert lora.lora_read_status() == lora.LORA_OK
        assert not torch.isnan(y).any() and not torch.isnan(su).any(), call
        # su comes from the same row-product launch either way
        assert torch.equal(su.view(torch.int16), p.su.view(torch.int16)), call
        if bitwise:
            assert torch.equal(y.view(torch.int16), p.y.view(torch.int16)), call
        else:
            assert G.rel_fro(G.host_f64(y), G.host_f64(p.y)) <= G.TOL_Y, call
        assert G.rel_fro(G.host_f64(y), y_want) <= G.TOL_Y, call
        assert G.rel_fro(G.host_f64(su), s * u) <= G.TOL_SU, call


def test_noalloc_rejects_shapes_beyond_its_scratch():
    # 16384 tokens x d_in 8192 at rank 64 needs far more than the fixed array
    T, K, N, r = 16384, 8192, 64, 64
    st = lora.make_shape(T, K, N, r, 2.0)
    small = torch.zeros(256, dtype=torch.bfloat16, device="cuda")
    y = torch.full((256,), float("nan"), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd_noalloc(st, small, small, small, small, y, None)
    assert e.value.code == lora.LORA_ESCRATCH
    # argument errors come first, as in lora_linear_fwd
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd_noalloc(st, small, small, None, small, y, None)
    assert e.value.code == lora.LORA_ENULL
    torch.cuda.synchronize()
    assert torch.isnan(y).all(), "a rejected call must enqueue nothing"
    assert np.isnan(G.host_f64(y)).all()
