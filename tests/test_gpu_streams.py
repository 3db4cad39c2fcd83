"""GPU tests of the two-stream schedule of calls with a backward (the
backward's rank-r work on a side stream joined by events): a call captured
into a CUDA graph and replayed, and calls from two host threads on their own
streams at the same time, give bit-identical results to the plain call; with
the side stream switched off (LORA_OVERLAP=0) the same call runs every step
on one stream and still matches the oracle."""
import os
import subprocess
import sys
import threading

import pytest
import torch

from paper_2606_19528_gb300 import lora, workloads
from tests import gpu_util as G
from tests.test_gpu_parity import build_layer

pytestmark = pytest.mark.gpu

OUTS = ("y", "su", "dx", "dA", "dB")


def snapshot(ps):
    return [{n: getattr(p, n).clone() for n in OUTS} for p in ps]


def same(a, b):
    for pa, pb in zip(a, b):
        for n in OUTS:
            x, y = pa[n], pb[n]
            if x.dtype == torch.bfloat16:
                x, y = x.view(torch.int16), y.view(torch.int16)
            if not torch.equal(x, y):
                return n
    return None


def fill_nan(ps):
    for p in ps:
        for n in OUTS:
            getattr(p, n).fill_(float("nan"))


def test_graph_capture_of_a_two_stream_call():
    wl = workloads.llama_sweep(256, 16)
    ps = build_layer(wl, seed=5)
    projs = [p.proj() for p in ps]
    ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_FWD_BWD))
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):  # capture needs a stream other than the legacy default
        lora.lora_stack_step(projs, lora.LORA_FWD_BWD, ws, ws.numel(), side)
    torch.cuda.synchronize()
    want = snapshot(ps)
    fill_nan(ps)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        lora.lora_stack_step(projs, lora.LORA_FWD_BWD, ws, ws.numel(), side)
    torch.cuda.synchronize()
    fill_nan(ps)  # capture records, it does not run
    g.replay()
    g.replay()
    torch.cuda.synchronize()
    assert same(snapshot(ps), want) is None
    assert lora.lora_read_status() == lora.LORA_OK


def test_two_host_threads_at_once():
    wl = workloads.llama_sweep(256, 16)
    layers = [build_layer(wl, seed=7 + t) for t in range(2)]
    wants = []
    for ps in layers:
        G.run_stack(ps)
        torch.cuda.synchronize()
        wants.append(snapshot(ps))
        fill_nan(ps)
    errors = []

    def work(ps):
        try:
            st = torch.cuda.Stream()
            projs = [p.proj() for p in ps]
            ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_FWD_BWD))
            for _ in range(3):
                lora.lora_stack_step(projs, lora.LORA_FWD_BWD, ws, ws.numel(), st)
            st.synchronize()
        except Exception as e:  # reported below
            errors.append(e)

    threads = [threading.Thread(target=work, args=(ps,)) for ps in layers]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    for ps, want in zip(layers, wants):
        assert same(snapshot(ps), want) is None


def test_graph_capture_of_a_backward_only_call():
    """A backward-only call also forks: sv on the caller's stream, then dA (and
    dB) on the side stream beside the dx contraction.  Captured and replayed,
    it matches the plain call bit for bit."""
    wl = workloads.llama_sweep(256, 16)
    ps = build_layer(wl, seed=9)
    projs = [p.proj() for p in ps]
    ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_FWD_BWD))
    side = torch.cuda.Stream()
    with torch.cuda.stream(side):
        lora.lora_stack_step(projs, lora.LORA_FWD, ws, ws.numel(), side)
        lora.lora_stack_step(projs, lora.LORA_BWD, ws, ws.numel(), side)
    torch.cuda.synchronize()
    want = snapshot(ps)
    bwd_outs = ("dx", "dA", "dB")
    for p in ps:
        for n in bwd_outs:
            getattr(p, n).fill_(float("nan"))
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        lora.lora_stack_step(projs, lora.LORA_BWD, ws, ws.numel(), side)
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    assert same(snapshot(ps), want) is None
    assert lora.lora_read_status() == lora.LORA_OK


ONE_STREAM = r"""
import sys
from paper_2606_19528_gb300 import lora, workloads
from tests import gpu_util as G
from tests.test_gpu_parity import build_layer, check_full
wl = workloads.llama_sweep(256, 16)
ps = build_layer(wl, seed=7)
G.run_stack(ps)
for p in ps:
    check_full(p)
print("one-stream call ok")
"""


def test_forward_and_backward_call_without_the_side_stream():
    """LORA_OVERLAP=0 (read once per process, hence a child process): the
    backward's rank-r work runs on the call's stream after the forward, on
    every SM; every output of the Llama-shaped layer at T = 256 against the
    oracle."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, LORA_OVERLAP="0")
    r = subprocess.run([sys.executable, "-c", ONE_STREAM], cwd=root, env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "one-stream call ok" in r.stdout
