"""GPU parity of the 4-bit base-weight path (Algorithm 1, on-the-fly
dequantization W = s * W_q + b inside the fused contractions) through the C
ABI, against the fp64 oracle on the same seeded codes, parameters and bf16
activations.  Tolerances as for bf16 weights (the dequantized element is
rounded to bf16 once before the tensor core uses it); exact where the
arithmetic is exact."""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2606_19528_gb300 import lora, synth, workloads
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


class DevQ4Proj(G.DevProj):
    """A projection whose base weight is given as 4-bit codes and (s, b) pairs."""

    def __init__(self, x, codes, params, A, B, dy, s, share_x=None):
        sb = synth.bf16_bits_to_f64(params)
        self.W64 = oracle.dequant_q4(codes, sb[..., 0], sb[..., 1])
        W_bits = synth.to_bf16_bits(self.W64)  # exact s q + b rounded once, as the kernels do
        super().__init__(x, W_bits, A, B, dy, s, share_x=share_x)
        self.codes = torch.from_numpy(np.ascontiguousarray(codes)).to("cuda")
        self.params = G.dev_bf16(params)
        self.Wq = lora.make_q4(self.codes, self.params)

    def proj(self, with_dx=True):
        return lora.make_proj(self.shape, x=self.x, A=self.A, B=self.B, dy=self.dy, y=self.y, su=self.su,
                              dx=self.dx if with_dx else None, dA=self.dA, dB=self.dB, Wq=self.Wq)


def gen_q4_proj(cfg, idx, layer, T, K, N, r, s, group=None, seed=0, share_x=None):
    x = synth.gen_x(seed, cfg, idx if group is None else group, layer, T, K)
    codes, params = synth.gen_Wq(seed, cfg, idx, layer, N, K)
    A = synth.gen_A(seed, cfg, idx, layer, r, K)
    B = synth.gen_B(seed, cfg, idx, layer, N, r)
    dy = synth.gen_dy(seed, cfg, idx, layer, T, N)
    return DevQ4Proj(x, codes, params, A, B, dy, s, share_x=share_x)


def run_q4_single(p: DevQ4Proj, with_dx=True):
    st = p.shape
    ws = G.workspace(lora.lora_workspace_size(st, lora.LORA_FWD_BWD))
    lora.lora_linear_fwd_q4(st, p.x, p.Wq, p.A, p.B, p.y, p.su, ws, ws.numel())
    lora.lora_linear_bwd_q4(st, p.dy, p.x, p.Wq, p.A, p.B, p.su, p.dx if with_dx else None, p.dA, p.dB, ws,
                            ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK


def check_q4_full(p: DevQ4Proj):
    x, A, B, dy = (p.f64(k) for k in ("x", "A", "B", "dy"))
    y, u = oracle.lora_forward(x, p.W64, A, B, p.s)
    dx, dA, dB, _ = oracle.lora_backward(dy, x, p.W64, A, B, p.s)
    errs = {"y": G.rel_fro(G.host_f64(p.y), y), "su": G.rel_fro(G.host_f64(p.su), p.s * u),
            "dx": G.rel_fro(G.host_f64(p.dx), dx), "dA": G.rel_fro(G.host_f64(p.dA), dA),
            "dB": G.rel_fro(G.host_f64(p.dB), dB)}
    for k, v in errs.items():
        assert v <= (G.TOL_GRAD if k in ("dA", "dB") else G.TOL_Y), (k, errs)
    return errs


def test_q4_handworked_exact():
    """The hand-worked dequantization (2 rows x 128 columns) embedded in a
    T = 8, d_in = 256, d_out = 8, r = 1 problem with A = B = 0 (zero codes and
    (s, b) = (0, 0) elsewhere): y = x W^T and dx = dy W (dy = unit rows, so dx
    reads back whole rows of W) are exact."""
    with open(os.path.join(GOLDEN, "q4_dequant_handworked_N2_K128.json")) as f:
        g = json.load(f)
    T, K, N, r = 8, 256, 8, 1
    codes = np.zeros((N, K // 2), dtype=np.uint8)
    codes[:2, :64] = np.array(g["codes"], dtype=np.uint8)
    s = np.zeros((N, K // 64))
    b = np.zeros((N, K // 64))
    s[:2, :2], b[:2, :2] = np.array(g["s"]), np.array(g["b"])
    params = np.stack([synth.to_bf16_bits(s), synth.to_bf16_bits(b)], axis=-1)
    x = np.zeros((T, K))
    x[:2, :128] = np.array(g["x"])
    dy = np.zeros((T, N))
    dy[0, 0] = dy[1, 1] = 1.0
    z = np.zeros
    p = DevQ4Proj(synth.to_bf16_bits(x), codes, params, synth.to_bf16_bits(z((r, K))),
                  synth.to_bf16_bits(z((N, r))), synth.to_bf16_bits(dy), 1.0)
    run_q4_single(p)
    y = G.host_f64(p.y)
    assert np.array_equal(y[:2, :2], np.array(g["y"])), y[:2, :2]
    assert np.array_equal(y[2:], np.zeros((T - 2, N))) and np.array_equal(y[:, 2:], np.zeros((T, N - 2)))
    dx = G.host_f64(p.dx)
    W = np.array(g["W"])
    assert np.array_equal(dx[:2, :128], W), dx[:2, :128]
    assert np.array_equal(dx[:2, 128:], np.zeros((2, 128)))
    assert np.array_equal(G.host_f64(p.dA), np.zeros((r, K)))


Q4_SHAPES = [(256, 256, 256, 16), (384, 512, 320, 8), (200, 768, 1024, 24), (136, 1024, 72, 3), (512, 3072, 1024, 16)]


@pytest.mark.parametrize("T,K,N,r", Q4_SHAPES, ids=[f"T{T}_K{K}_N{N}_r{r}" for T, K, N, r in Q4_SHAPES])
def test_q4_single_parity(T, K, N, r):
    p = gen_q4_proj(20, 0, 0, T, K, N, r, 2.0)
    run_q4_single(p)
    check_q4_full(p)


def test_q4_equals_bf16_path_on_dequantized_weight():
    """The tensor core sees the same bf16 operands either way (bf16(s q + b),
    rounded once), and the 4-bit kernel keeps the bf16 kernel's tile order and
    contraction order: y, su and dx agree bit for bit.  The shape has 80
    output tiles either way, so neither path cuts its contractions (the bf16
    path cuts few-tile contractions between cluster pairs, the 4-bit path into
    fp32 partials).  dA and dB come from the rank-r kernels on the side stream,
    whose width follows the contraction beside it (4-bit contractions are
    weighted as slower), so their sums over 2048 tokens may be cut
    differently: equal to the fp32 rounding of such sums (~1e-6 relative)."""
    T, K, N, r = 2048, 5120, 5120, 16
    p = gen_q4_proj(21, 0, 0, T, K, N, r, 2.0)
    run_q4_single(p)
    q = G.DevProj(*(p.bits[k] for k in ("x", "W", "A", "B", "dy")), p.s)
    G.run_single(q)
    for n in ("y", "su", "dx"):
        assert torch.equal(getattr(p, n).view(torch.int16), getattr(q, n).view(torch.int16)), n
    for n in ("dA", "dB"):
        assert G.rel_fro(G.host_f64(getattr(p, n)), G.host_f64(getattr(q, n))) < 1e-5, n


def test_q4_layer_stack_mixed():
    """A Llama-3.2-3B-shaped layer at T = 512 with q, k, v, gate, up and down
    in 4-bit form and o in bf16: one lora_stack_step launches both kernel
    variants; every projection against the oracle."""
    T, r, s = 512, 16, 2.0
    ps, xs = [], {}
    for i, pr in enumerate(workloads.llama_layer()):
        share = xs.get(pr.group)
        if pr.name == "o":
            x = synth.gen_x(0, 22, pr.group, 0, T, pr.d_in)
            W = synth.gen_W(0, 22, i, 0, pr.d_out, pr.d_in)
            A = synth.gen_A(0, 22, i, 0, r, pr.d_in)
            B = synth.gen_B(0, 22, i, 0, pr.d_out, r)
            dy = synth.gen_dy(0, 22, i, 0, T, pr.d_out)
            p = G.DevProj(x, W, A, B, dy, s, share_x=share)
            p.W64 = synth.bf16_bits_to_f64(W)
        else:
            p = gen_q4_proj(22, i, 0, T, pr.d_in, pr.d_out, r, s, group=pr.group, share_x=share)
        xs.setdefault(pr.group, p.x)
        ps.append(p)
    G.run_stack(ps)
    for p in ps:
        check_q4_full(p)  # every element of y, su, dx, dA and dB
        for t in (p.y, p.su, p.dx, p.dA, p.dB):
            assert not torch.isnan(t).any(), "an output element was never written"


def test_q4_llama_layer_T2048():
    """The 4-bit benchmark workload: the Llama-3.2-3B-shaped layer at
    T = 2048, r = 16 with every base weight in 4-bit form, one
    forward-and-backward call; every element against the fp64 oracle on the
    dequantized weights."""
    wl = workloads.llama_layer_T2048_q4()
    ps, xs = [], {}
    for i, pr in enumerate(wl.projs):
        p = gen_q4_proj(wl.cfg, i, 0, wl.T, pr.d_in, pr.d_out, wl.rank, wl.scale, group=pr.group,
                        share_x=xs.get(pr.group))
        xs.setdefault(pr.group, p.x)
        ps.append(p)
    G.run_stack(ps)
    for p in ps:
        check_q4_full(p)


def test_q4_argument_errors():
    T, K, N, r = 64, 256, 64, 8
    p = gen_q4_proj(23, 0, 0, T, K, N, r, 2.0)
    ws = G.workspace(lora.lora_workspace_size(p.shape, lora.LORA_FWD_BWD))
    bad_K = lora.make_shape(T, 128, N, r, 2.0)  # d_in not a multiple of 256
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd_q4(bad_K, p.x, p.Wq, p.A, p.B, p.y, p.su, ws, ws.numel())
    assert e.value.code == lora.LORA_EINVAL
    both = lora.make_proj(p.shape, x=p.x, W=p.W, A=p.A, B=p.B, y=p.y, su=p.su, Wq=p.Wq)
    with pytest.raises(lora.LoraError) as e:
        lora.lora_stack_step([both], lora.LORA_FWD, ws, ws.numel())
    assert e.value.code == lora.LORA_EINVAL
    half = lora.make_q4(p.codes, None)
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd_q4(p.shape, p.x, half, p.A, p.B, p.y, p.su, ws, ws.numel())
    assert e.value.code == lora.LORA_ENULL
    torch.cuda.synchronize()
    assert torch.isnan(p.y).all(), "a rejected call must enqueue nothing"
