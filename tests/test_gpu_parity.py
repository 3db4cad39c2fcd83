"""GPU parity: the CUDA path, called through the C ABI, against the fp64 oracle
on the same seeded bf16 inputs.  Tolerances: relative Frobenius error
<= 5e-3 for y, su and dx, <= 1e-2 for dA and dB; exact where the arithmetic
is exact (small integers, B = 0)."""
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


def gen_proj(cfg, idx, layer, T, K, N, r, s, group=None, zero_B=False, seed=0):
    x = synth.gen_x(seed, cfg, idx if group is None else group, layer, T, K)
    W = synth.gen_W(seed, cfg, idx, layer, N, K)
    A = synth.gen_A(seed, cfg, idx, layer, r, K)
    B = synth.gen_B(seed, cfg, idx, layer, N, r, zero=zero_B)
    dy = synth.gen_dy(seed, cfg, idx, layer, T, N)
    return x, W, A, B, dy


def check_full(p: G.DevProj, with_dx=True):
    x, W, A, B, dy = (p.f64(k) for k in ("x", "W", "A", "B", "dy"))
    y, u = oracle.lora_forward(x, W, A, B, p.s)
    dx, dA, dB, _ = oracle.lora_backward(dy, x, W, A, B, p.s)
    errs = {
        "y": G.rel_fro(G.host_f64(p.y), y),
        "su": G.rel_fro(G.host_f64(p.su), p.s * u),
        "dA": G.rel_fro(G.host_f64(p.dA), dA),
        "dB": G.rel_fro(G.host_f64(p.dB), dB),
    }
    if with_dx:
        errs["dx"] = G.rel_fro(G.host_f64(p.dx), dx)
    assert errs["y"] <= G.TOL_Y, errs
    assert errs["su"] <= G.TOL_SU, errs
    assert errs["dA"] <= G.TOL_GRAD, errs
    assert errs["dB"] <= G.TOL_GRAD, errs
    if with_dx:
        assert errs["dx"] <= G.TOL_DX, errs
    return errs


def check_sampled(p: G.DevProj, rows, with_dx=True):
    """Rows of y and dx computed one by one by the oracle; dA and dB in full."""
    x, W, A, B, dy = (p.f64(k) for k in ("x", "W", "A", "B", "dy"))
    y_rows = oracle.lora_forward_rows(rows, x, W, A, B, p.s)
    dA, dB = oracle.lora_adapter_grads(dy, x, A, B, p.s)
    su_rows = p.s * (x[rows] @ A.T)
    errs = {
        "y": G.rel_fro(G.host_f64(p.y)[rows], y_rows),
        "su": G.rel_fro(G.host_f64(p.su)[rows], su_rows),
        "dA": G.rel_fro(G.host_f64(p.dA), dA),
        "dB": G.rel_fro(G.host_f64(p.dB), dB),
    }
    if with_dx:
        dx_rows = oracle.lora_backward_dx_rows(rows, dy, W, A, B, p.s)
        errs["dx"] = G.rel_fro(G.host_f64(p.dx)[rows], dx_rows)
    for k, v in errs.items():
        tol = G.TOL_GRAD if k in ("dA", "dB") else G.TOL_Y
        assert v <= tol, (k, errs)
    for t in (p.y, p.su, p.dA, p.dB) + ((p.dx,) if with_dx else ()):
        assert not torch.isnan(t).any(), "an output element was never written"
    return errs


# --------------------------------------------------------------- exact cases

def test_handworked_example_exact():
    """The hand-worked integer example embedded in an 8 x 8 x 8 problem with
    r = 1 (zero padding elsewhere): every result is exact in bf16 / fp32."""
    with open(os.path.join(GOLDEN, "lora_handworked_T2_K3_N2_r1.json")) as f:
        g = json.load(f)
    T = K = N = 8
    r = 1

    def emb(name, rows, cols):
        a = np.zeros((rows, cols))
        v = np.array(g[name], dtype=np.float64)
        a[:v.shape[0], :v.shape[1]] = v
        return synth.to_bf16_bits(a)

    p = G.DevProj(emb("x", T, K), emb("W", N, K), emb("A", r, K), emb("B", N, r), emb("dy", T, N), g["s"])
    G.run_single(p)
    got = {"y": G.host_f64(p.y), "su": G.host_f64(p.su), "dx": G.host_f64(p.dx), "dA": G.host_f64(p.dA),
           "dB": G.host_f64(p.dB)}
    want = {"y": g["y"], "su": (np.array(g["u"]) * g["s"]).tolist(), "dx": g["dx"], "dA": g["dA"], "dB": g["dB"]}
    for k in want:
        w = np.array(want[k], dtype=np.float64)
        full = np.zeros_like(got[k])
        full[:w.shape[0], :w.shape[1]] = w
        assert np.array_equal(got[k], full), (k, got[k], full)


def test_single_small_T128():
    wl = workloads.single_small()
    pr = wl.projs[0]
    p = G.DevProj(*gen_proj(wl.cfg, 0, 0, wl.T, pr.d_in, pr.d_out, wl.rank, wl.scale), wl.scale)
    G.run_single(p)
    check_full(p)


def run_frozen(x_bits, W_bits, dy_bits):
    """The same contraction kernel with no adapter slab at all (rank 0: a
    frozen projection): y = x W^T and dx = dy W.  Returns (y, dx)."""
    T, K = x_bits.shape
    N = W_bits.shape[0]
    x, W, dy = G.dev_bf16(x_bits), G.dev_bf16(W_bits), G.dev_bf16(dy_bits)
    y = torch.full((T, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    dx = torch.full((T, K), float("nan"), dtype=torch.bfloat16, device="cuda")
    st = lora.make_shape(T, K, N, 0, 1.0)
    ws = G.workspace(lora.lora_workspace_size(st, lora.LORA_FWD_BWD))
    lora.lora_linear_fwd(st, x, W, None, None, y, None, ws, ws.numel())
    lora.lora_linear_bwd(st, dy, x, W, None, None, None, dx, None, None, ws, ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK
    return y, dx


# Shapes whose contractions run in one pass with and without the slab: a
# contraction with fewer output tiles than CTA pairs may be split along its
# depth, and how depends on that depth (K + r against K alone), which would
# change the fp32 summation order.  One 256 x 512 tile of 4-5 blocks never
# splits; 76 or more tiles never split.
B0_SHAPES = [(128, 256, 256), (2056, 4104, 4616)]


@pytest.mark.parametrize("T,K,N", B0_SHAPES, ids=[f"T{t}_K{k}_N{n}" for t, k, n in B0_SHAPES])
def test_init_invariant_B0(T, K, N):
    """B = 0 (LoRA initialisation): dA is exactly zero, and y and dx are bit
    for bit those of the same contraction with the adapter slab skipped
    (rank 0): the slab adds exact zeros to the fp32 accumulator.  Ranks 8 and
    16 (slabs of one 64-deep block, different fill) and a padded rank 3; the
    first shape is the single-projection workload with its B = 0 twin, the
    second has tails in every tile dimension."""
    wl = workloads.single_small(zero_B=True)
    x, W, _, _, dy = gen_proj(wl.cfg, 0, 0, T, K, N, 8, wl.scale, zero_B=True)
    y0, dx0 = run_frozen(x, W, dy)
    for r in (8, 16, 3):
        _, _, A, B, _ = gen_proj(wl.cfg, 0, 0, T, K, N, r, 16.0 / r, zero_B=True)
        p = G.DevProj(x, W, A, B, dy, 16.0 / r)
        G.run_single(p)
        assert not torch.any(p.dA != 0), "dA must be exactly 0 when B = 0"
        if r == 8 or T * K * N < 1e8:  # the oracle once per large shape
            check_full(p)
        assert torch.equal(p.y.view(torch.int16), y0.view(torch.int16)), r
        assert torch.equal(p.dx.view(torch.int16), dx0.view(torch.int16)), r


def test_frozen_projection_against_oracle():
    """Rank 0 is a frozen linear: y = x W^T and dx = dy W against the oracle
    (whose adapter terms are empty), ragged tiles in every dimension."""
    T, K, N = 264, 1032, 392
    x, W, _, _, dy = gen_proj(30, 0, 0, T, K, N, 1, 1.0)
    y, dx = run_frozen(x, W, dy)
    xf, Wf, dyf = (synth.bf16_bits_to_f64(b) for b in (x, W, dy))
    A0, B0 = np.zeros((0, K)), np.zeros((N, 0))
    y_want, _ = oracle.lora_forward(xf, Wf, A0, B0, 1.0)
    dx_want, _, _, _ = oracle.lora_backward(dyf, xf, Wf, A0, B0, 1.0)
    assert G.rel_fro(G.host_f64(y), y_want) <= G.TOL_Y
    assert G.rel_fro(G.host_f64(dx), dx_want) <= G.TOL_DX


# --------------------------------------------------------------- ragged shapes

RAGGED = [
    # T, K, N, r : tails in every tile dimension, minimal sizes, padded ranks
    (8, 8, 8, 1),
    (136, 200, 264, 24),
    (264, 72, 520, 4),
    (128, 320, 136, 72),
    (200, 136, 64, 128),
    (72, 1032, 392, 16),
    (384, 256, 768, 3),
]


@pytest.mark.parametrize("T,K,N,r", RAGGED, ids=[f"T{t}_K{k}_N{n}_r{r}" for t, k, n, r in RAGGED])
def test_ragged_shapes(T, K, N, r):
    s = 2.0
    p = G.DevProj(*gen_proj(7, r, T, T, K, N, r, s), s)
    G.run_single(p)
    check_full(p)


def test_forward_without_saved_su_and_backward_without_dx():
    T, K, N, r, s = 256, 512, 384, 16, 2.0
    bits = gen_proj(8, 0, 0, T, K, N, r, s)
    p = G.DevProj(*bits, s)
    G.run_single(p)
    q = G.DevProj(*bits, s)
    st = q.shape
    ws = G.workspace(lora.lora_workspace_size(st, lora.LORA_FWD_BWD))
    lora.lora_linear_fwd(st, q.x, q.W, q.A, q.B, q.y, None, ws, ws.numel())
    lora.lora_linear_bwd(st, q.dy, q.x, q.W, q.A, q.B, p.su, None, q.dA, q.dB, ws, ws.numel())
    torch.cuda.synchronize()
    assert torch.equal(p.y.view(torch.int16), q.y.view(torch.int16))
    assert torch.equal(p.dA, q.dA) and torch.equal(p.dB, q.dB)
    assert torch.isnan(q.dx).all(), "dx = NULL must leave dx untouched"


def test_deterministic():
    T, K, N, r, s = 512, 1024, 768, 16, 2.0
    bits = gen_proj(9, 0, 0, T, K, N, r, s)
    a, b = G.DevProj(*bits, s), G.DevProj(*bits, s)
    G.run_single(a)
    G.run_single(b)
    for n in ("y", "su", "dx"):
        assert torch.equal(getattr(a, n).view(torch.int16), getattr(b, n).view(torch.int16)), n
    assert torch.equal(a.dA, b.dA) and torch.equal(a.dB, b.dB)


# --------------------------------------------------------------- workloads

def test_llama_q_T512():
    wl = workloads.llama_q()
    pr = wl.projs[0]
    p = G.DevProj(*gen_proj(wl.cfg, 0, 0, wl.T, pr.d_in, pr.d_out, wl.rank, wl.scale), wl.scale)
    G.run_single(p)
    check_full(p)


def build_layer(wl, layer=0, seed=0):
    xs = {}
    ps = []
    for i, pr in enumerate(wl.projs):
        x, W, A, B, dy = gen_proj(wl.cfg, i, layer, wl.T, pr.d_in, pr.d_out, wl.rank, wl.scale, group=pr.group,
                                  seed=seed)
        share = xs.get(pr.group)
        p = G.DevProj(x, W, A, B, dy, wl.scale, share_x=share)
        xs.setdefault(pr.group, p.x)
        ps.append(p)
    return ps


@pytest.mark.parametrize("name", ["llama_layer", "qwen_layer"])
def test_layer_stack(name):
    """The Llama-3.2-3B-shaped layer at T = 2048, r = 16 and the
    Qwen-2.5-3B-shaped layer at T = 4096, r = 64, in the launch
    configuration the benchmark times (one forward-and-backward call, side
    stream): every element of y, su, dx, dA and dB against the fp64 oracle."""
    wl = workloads.BY_NAME[name]()
    ps = build_layer(wl)
    G.run_stack(ps)
    for p in ps:
        check_full(p)
        for t in (p.y, p.su, p.dx, p.dA, p.dB):
            assert not torch.isnan(t).any(), "an output element was never written"


def test_layer_adapting_q_and_v_only():
    """The paper's own setting: adapters on q and v only (hyper-parameter
    table), the other five projections frozen (rank 0) but still on the
    backward path through dx.  One call over the Llama-shaped layer at
    T = 512: the adapted projections against the oracle in full, the frozen
    ones as y = x W^T and dx = dy W, and dA / dB of the frozen ones untouched."""
    T, r, s = 512, 16, 2.0
    ps, xs, frozen = [], {}, []
    for i, pr in enumerate(workloads.llama_layer()):
        rr = r if pr.name in ("q", "v") else 0
        bits = gen_proj(31, i, 0, T, pr.d_in, pr.d_out, max(rr, 1), s, group=pr.group)
        if rr == 0:
            bits = (bits[0], bits[1], np.zeros((0, pr.d_in), np.uint16), np.zeros((pr.d_out, 0), np.uint16),
                    bits[4])
        p = G.DevProj(*bits, s, share_x=xs.get(pr.group))
        xs.setdefault(pr.group, p.x)
        ps.append(p)
        frozen.append(rr == 0)
    projs = []
    for p, fz in zip(ps, frozen):
        if fz:
            projs.append(lora.make_proj(p.shape, x=p.x, W=p.W, dy=p.dy, y=p.y, dx=p.dx))
        else:
            projs.append(p.proj())
    ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_FWD_BWD))
    lora.lora_stack_step(projs, lora.LORA_FWD_BWD, ws, ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK
    for p, fz in zip(ps, frozen):
        if not fz:
            check_full(p)
            continue
        x, W, dy = (p.f64(k) for k in ("x", "W", "dy"))
        assert G.rel_fro(G.host_f64(p.y), x @ W.T) <= G.TOL_Y
        assert G.rel_fro(G.host_f64(p.dx), dy @ W) <= G.TOL_DX


def test_stack_equals_single_calls():
    """The grouped launches compute su exactly as single calls do; y and dx
    agree up to the bf16 rounding of differently ordered fp32 sums (with few
    output tiles the contractions are split, and how depends on the launch's
    problems), dA and dB (whose token reduction is split by launch) to fp32
    rounding; a repeated stack call is bit-identical."""
    wl = workloads.llama_sweep(256, 16)
    ps = build_layer(wl, seed=3)
    G.run_stack(ps)
    first = [(p.dA.clone(), p.dB.clone(), p.y.clone()) for p in ps]
    G.run_stack(ps)
    for p, (dA, dB, y) in zip(ps, first):
        assert torch.equal(p.dA, dA) and torch.equal(p.dB, dB) and torch.equal(p.y.view(torch.int16), y.view(torch.int16))
    for i, pr in enumerate(wl.projs):
        q = G.DevProj(*(ps[i].bits[k] for k in ("x", "W", "A", "B", "dy")), wl.scale)
        G.run_single(q)
        assert torch.equal(q.su.view(torch.int16), ps[i].su.view(torch.int16)), (pr.name, "su")
        for n in ("y", "dx"):
            assert G.rel_fro(G.host_f64(getattr(q, n)), G.host_f64(getattr(ps[i], n))) < 2e-3, (pr.name, n)
        assert G.rel_fro(G.host_f64(q.dA), G.host_f64(ps[i].dA)) < 1e-6, pr.name
        assert G.rel_fro(G.host_f64(q.dB), G.host_f64(ps[i].dB)) < 1e-6, pr.name


def test_stack_mixed_ranks_fused_and_two_pass():
    """One call whose projections take both backward paths over dy: r <= 16
    the fused pass (sv and dB in one read), r > 16 the two separate passes,
    sharing one partial arena in turn; ragged T and N, projections sharing x.
    Every output against the oracle; the backward-only call (all SMs, other
    cuts) agrees with the two-stream call to fp32 rounding."""
    T, s = 648, 2.0
    shapes = [(520, 392, 16), (520, 136, 32), (520, 264, 3), (392, 520, 64), (136, 1032, 8)]
    groups = [0, 0, 0, 1, 2]
    ps, xs = [], {}
    for i, ((K, N, r), g) in enumerate(zip(shapes, groups)):
        bits = gen_proj(21, i, 0, T, K, N, r, s, group=g)
        p = G.DevProj(*bits, s, share_x=xs.get(g))
        xs.setdefault(g, p.x)
        ps.append(p)
    G.run_stack(ps)
    for p in ps:
        check_full(p)
    first = [(p.dA.clone(), p.dB.clone(), p.dx.clone()) for p in ps]
    G.run_stack(ps, lora.LORA_FWD)
    G.run_stack(ps, lora.LORA_BWD)
    for p, (dA, dB, dx) in zip(ps, first):
        assert G.rel_fro(G.host_f64(p.dA), G.host_f64(dA)) < 1e-6
        assert G.rel_fro(G.host_f64(p.dB), G.host_f64(dB)) < 1e-6
        assert G.rel_fro(G.host_f64(p.dx), G.host_f64(dx)) < 2e-3


SWEEP = [(T, r) for T in workloads.SWEEP_TOKENS for r in workloads.SWEEP_RANKS]


@pytest.mark.parametrize("T,r", SWEEP, ids=[f"T{T}_r{r}" for T, r in SWEEP])
def test_rank_token_sweep(T, r):
    wl = workloads.llama_sweep(T, r)
    ps = build_layer(wl)
    G.run_stack(ps)
    rows = G.sample_rows(T, 32, T + r)
    for p in ps:
        check_sampled(p, rows)
    del ps
    torch.cuda.empty_cache()


def test_stack28_forward_all_then_backward_all():
    """28 layers: forward of every layer first (saving su), then backward of
    every layer in reverse order from the stored inputs."""
    wl = workloads.llama_stack28()
    layers = [build_layer(wl, layer=l) for l in range(wl.layers)]
    for ps in layers:
        projs = [p.proj() for p in ps]
        ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_FWD))
        lora.lora_stack_step(projs, lora.LORA_FWD, ws, ws.numel())
    for ps in reversed(layers):
        projs = [p.proj() for p in ps]
        ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_BWD))
        lora.lora_stack_step(projs, lora.LORA_BWD, ws, ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK
    rows = G.sample_rows(wl.T, 8, 5)
    for l, ps in enumerate(layers):
        for p in ps:
            check_sampled(p, rows)


# --------------------------------------------------------------- argument errors on the device path

def test_argument_errors():
    T, K, N, r, s = 128, 256, 256, 8, 2.0
    p = G.DevProj(*gen_proj(0, 0, 0, T, K, N, r, s), s)
    st = p.shape
    need = lora.lora_workspace_size(st, lora.LORA_FWD)
    ws = G.workspace(need + 512)
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd(st, p.x, p.W, p.A, p.B, p.y, p.su, ws, need - 1)
    assert e.value.code == lora.LORA_EWORKSPACE
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd(st, p.x.data_ptr() + 2, p.W, p.A, p.B, p.y, p.su, ws, need)
    assert e.value.code == lora.LORA_EALIGN
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd(st, p.x, p.W, p.A, p.B, p.y, p.su, ws.data_ptr() + 16, need)
    assert e.value.code == lora.LORA_EALIGN
    for bad in (lora.make_shape(12, K, N, r, s), lora.make_shape(T, K, N, -1, s), lora.make_shape(T, K, N, 129, s),
                lora.make_shape(T, K, N, r, float("inf"))):
        with pytest.raises(lora.LoraError) as e:
            lora.lora_linear_fwd(bad, p.x, p.W, p.A, p.B, p.y, p.su, ws, need)
        assert e.value.code == lora.LORA_EINVAL
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_bwd(st, p.dy, p.x, p.W, p.A, p.B, None, p.dx, p.dA, p.dB, ws, need)
    assert e.value.code == lora.LORA_ENULL
    assert lora.lora_last_error() == lora.LORA_ENULL
    lora.lora_linear_fwd(st, p.x, p.W, p.A, p.B, p.y, p.su, ws, need)
    assert lora.lora_last_error() == lora.LORA_OK
    torch.cuda.synchronize()
    p.y.fill_(float("nan"))
    with pytest.raises(lora.LoraError) as e:
        lora.lora_linear_fwd(st, p.x, p.W, None, p.B, p.y, p.su, ws, need)  # rank 8 needs A
    assert e.value.code == lora.LORA_ENULL
    torch.cuda.synchronize()
    assert torch.isnan(p.y).all(), "a rejected call must enqueue nothing"


# --------------------------------------------------------------- failure detection

def test_bounded_wait_expires_and_context_survives():
    """A wait on a barrier nothing arrives on gives up after its limit, the
    status word says LORA_ETIMEOUT, and the next call runs normally."""
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK
    lora.lora_wait_selftest(2_000_000)  # 2 ms
    assert lora.lora_read_status(reset=True) == lora.LORA_ETIMEOUT
    assert lora.lora_read_status() == lora.LORA_OK
    s = 2.0
    p = G.DevProj(*gen_proj(0, 7, 0, 128, 256, 256, 8, s), s)
    G.run_single(p)
    check_full(p)


# --------------------------------------------------------------- data-parallel sharding identity

def test_token_shards_sum_to_the_unsharded_gradients():
    """The token sharding of a data-parallel step, run one shard after the
    other on one GPU: each shard's y, su and dx are the matching rows of the
    unsharded call's (within rounding: the contractions may split
    differently), and the shards' dA and dB summed through the all-reduce
    hook (here a local sum of the shards' buffers) equal the unsharded
    gradients up to the bf16 rounding of sv and su (their fp32 sums are cut
    differently for a shard, so an element may round to the neighbouring
    bf16 value, ~1e-5 relative in dA and dB) and fp32 rounding; both against
    the oracle."""
    from paper_2606_19528_gb300 import shard
    T, K, N, r, s, world = 1032, 1024, 768, 16, 2.0, 3
    bits = gen_proj(32, 0, 0, T, K, N, r, s)
    full = G.DevProj(*bits, s)
    G.run_single(full)
    check_full(full)
    x, W, A, B, dy = bits
    parts = []
    for rank in range(world):
        t0, t1 = shard.token_slice(T, rank, world)
        p = G.DevProj(x[t0:t1], W, A, B, dy[t0:t1], s)
        G.run_single(p)
        for n in ("y", "su", "dx"):
            assert G.rel_fro(G.host_f64(getattr(p, n)), G.host_f64(getattr(full, n))[t0:t1]) <= 2e-3, (rank, n)
        parts.append(p)
    grads = [[p.dA.clone(), p.dB.clone()] for p in parts]

    def hook_for(rank):
        def hook(buf):  # sums the packed buffers of every shard, as an all-reduce would
            packed = [torch.cat([g.reshape(-1) for g in gs]) for gs in grads]
            buf.copy_(torch.stack(packed).sum(0))
        return hook

    summed = [[g.clone() for g in gs] for gs in grads]
    for rank in range(world):
        shard.sum_adapter_grads(summed[rank], hook_for(rank))
    for rank in range(world):
        assert G.rel_fro(G.host_f64(summed[rank][0]), G.host_f64(full.dA)) < 1e-4
        assert G.rel_fro(G.host_f64(summed[rank][1]), G.host_f64(full.dB)) < 1e-4
        assert torch.equal(summed[rank][0], summed[0][0]) and torch.equal(summed[rank][1], summed[0][1])
    dA, dB = oracle.lora_adapter_grads(full.f64("dy"), full.f64("x"), full.f64("A"), full.f64("B"), s)
    assert G.rel_fro(G.host_f64(summed[0][0]), dA) <= G.TOL_GRAD
    assert G.rel_fro(G.host_f64(summed[0][1]), dB) <= G.TOL_GRAD


# --------------------------------------------------------------- contractions with few output tiles

# Shapes whose forward and backward contractions have few output tiles, so that each 256 x 256 tile is
# shared by the two CTA pairs of a cluster (halves of the contraction summed in distributed shared
# memory): ragged tokens and columns, the smallest depth the library cuts this way (8 blocks: the
# backward of the first shape, 392 + 24 deep), a rank that pads, and a frozen projection.
CS_SHAPES = [(264, 520, 392, 24), (136, 1032, 520, 3), (512, 3072, 3072, 16), (392, 2056, 1544, 0)]


@pytest.mark.parametrize("T,K,N,r", CS_SHAPES, ids=[f"T{t}_K{k}_N{n}_r{r}" for t, k, n, r in CS_SHAPES])
def test_few_tile_contractions(T, K, N, r):
    """Every output against the oracle, and a second call bit for bit equal to the first (the two halves
    are added in one fp32 operation, whichever pair adds them)."""
    s = 2.0
    if r == 0:
        x, W, _, _, dy = gen_proj(33, 0, 0, T, K, N, 1, s)
        y, dx = run_frozen(x, W, dy)
        xf, Wf, dyf = (synth.bf16_bits_to_f64(b) for b in (x, W, dy))
        assert G.rel_fro(G.host_f64(y), xf @ Wf.T) <= G.TOL_Y
        assert G.rel_fro(G.host_f64(dx), dyf @ Wf) <= G.TOL_DX
        y2, dx2 = run_frozen(x, W, dy)
        assert torch.equal(y.view(torch.int16), y2.view(torch.int16))
        assert torch.equal(dx.view(torch.int16), dx2.view(torch.int16))
        return
    bits = gen_proj(33, r, 0, T, K, N, r, s)
    p = G.DevProj(*bits, s)
    G.run_single(p)
    check_full(p)
    q = G.DevProj(*bits, s)
    G.run_single(q)
    for n in ("y", "su", "dx"):
        assert torch.equal(getattr(p, n).view(torch.int16), getattr(q, n).view(torch.int16)), n
    assert torch.equal(p.dA, q.dA) and torch.equal(p.dB, q.dB)
