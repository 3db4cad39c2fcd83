"""CPU tests of the data-parallel token sharding (host logic): the slices
cover the tokens exactly, and the sharding identity holds through the
all-reduce hook among world-size-2 gloo ranks:

    sum over ranks of dA(tokens of the rank) = dA(all tokens), same for dB,

because dA = s (dy B)^T x and dB = s dy^T (x A^T) are sums over tokens.
Each rank computes its slice's gradients with the fp64 oracle (rounded to
fp32, as the library returns them); no GPU and no collective on a device."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2606_19528_gb300 import shard, synth


@pytest.mark.parametrize("T,world", [(2048, 2), (520, 3), (8, 4), (4096, 8), (0, 2)])
def test_token_slices_cover_the_tokens(T, world):
    sl = [shard.token_slice(T, r, world) for r in range(world)]
    assert sl[0][0] == 0 and sl[-1][1] == T
    for (a0, a1), (b0, b1) in zip(sl, sl[1:]):
        assert a1 == b0
    lens = [b - a for a, b in sl]
    assert all(a % 8 == 0 and b % 8 == 0 for a, b in sl)
    assert max(lens) - min(lens) <= 8


def test_token_slice_rejects_bad_arguments():
    with pytest.raises(ValueError):
        shard.token_slice(12, 0, 2)
    with pytest.raises(ValueError):
        shard.token_slice(16, 2, 2)


def _inputs(T, K, N, r):
    f = synth.bf16_bits_to_f64
    return (f(synth.gen_x(0, 40, 0, 0, T, K)), f(synth.gen_A(0, 40, 0, 0, r, K)), f(synth.gen_B(0, 40, 0, 0, N, r)),
            f(synth.gen_dy(0, 40, 0, 0, T, N)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    T, K, N, r, s = 520, 96, 72, 8, 2.0
    x, A, B, dy = _inputs(T, K, N, r)
    t0, t1 = shard.token_slice(T, rank, world)
    dA, dB = oracle.lora_adapter_grads(dy[t0:t1], x[t0:t1], A, B, s)
    g = [torch.from_numpy(dA.astype(np.float32)), torch.from_numpy(dB.astype(np.float32))]
    calls = []

    def hook(buf):  # the pluggable exchange: here gloo's all-reduce, counted
        calls.append(buf.numel())
        dist.all_reduce(buf, op=dist.ReduceOp.SUM)

    shard.sum_adapter_grads(g, hook)
    q.put((rank, g[0].numpy(), g[1].numpy(), calls))
    dist.destroy_process_group()


def test_sharding_identity_through_the_allreduce_hook_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = {}
    for _ in range(2):
        rank, dA, dB, calls = q.get(timeout=120)
        got[rank] = (dA, dB, calls)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    T, K, N, r, s = 520, 96, 72, 8, 2.0
    x, A, B, dy = _inputs(T, K, N, r)
    dA, dB = oracle.lora_adapter_grads(dy, x, A, B, s)
    for rank in (0, 1):
        gA, gB, calls = got[rank]
        assert calls == [r * K + N * r], "one packed exchange per step"
        # the sum of two fp32-rounded halves: within a few fp32 ulps of the whole
        assert np.max(np.abs(gA - dA)) <= 4e-7 * np.max(np.abs(dA))
        assert np.max(np.abs(gB - dB)) <= 4e-7 * np.max(np.abs(dB))
    assert np.array_equal(got[0][0], got[1][0]) and np.array_equal(got[0][1], got[1][1])


def test_sum_adapter_grads_without_ranks_is_the_identity():
    g = [torch.ones(3, 4), torch.full((2,), 2.0)]
    shard.sum_adapter_grads(g, lambda buf: None)
    assert torch.equal(g[0], torch.ones(3, 4)) and torch.equal(g[1], torch.full((2,), 2.0))
    with pytest.raises(TypeError):
        shard.sum_adapter_grads([torch.ones(2, dtype=torch.float64)], lambda buf: None)
