"""GPU tests of the checkpointed stack schedule (Algorithm 2: every layer's
forward without saving anything, then from the last layer back a re-forward
that keeps su in the workspace and the backward), through the C ABI."""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_19528_gb300 import lora, workloads
from tests import gpu_util as G
from tests.test_gpu_parity import build_layer

pytestmark = pytest.mark.gpu


def _outputs(ps):
    return [(p.y.view(torch.int16).clone(), p.dx.view(torch.int16).clone(), p.dA.clone(), p.dB.clone()) for p in ps]


def test_ckpt_equals_saved_schedule_and_oracle():
    """Four Llama-3.2-3B-shaped layers at T = 256: the checkpointed schedule
    gives bit for bit what forward-all-then-backward-all with saved su gives
    (the re-forward recomputes the same su with the same kernels), and the
    oracle agrees on sampled rows of every layer."""
    wl = workloads.llama_sweep(256, 16)
    L = 4
    layers = [build_layer(wl, layer=l, seed=5) for l in range(L)]
    # saved-activation schedule
    for ps in layers:
        projs = [p.proj() for p in ps]
        ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_FWD))
        lora.lora_stack_step(projs, lora.LORA_FWD, ws, ws.numel())
    for ps in reversed(layers):
        projs = [p.proj() for p in ps]
        ws = G.workspace(lora.lora_stack_workspace_size(projs, lora.LORA_BWD))
        lora.lora_stack_step(projs, lora.LORA_BWD, ws, ws.numel())
    torch.cuda.synchronize()
    saved = [_outputs(ps) for ps in layers]
    for ps in layers:
        for p in ps:
            for t in (p.y, p.dx, p.dA, p.dB):
                t.fill_(float("nan"))
    # checkpointed schedule
    projs = [[p.proj() for p in ps] for ps in layers]
    ws = G.workspace(lora.lora_stack_ckpt_workspace_size(projs))
    lora.lora_stack_ckpt(projs, ws, ws.numel())
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK
    for l, ps in enumerate(layers):
        for p, (y, dx, dA, dB) in zip(ps, saved[l]):
            assert torch.equal(p.y.view(torch.int16), y), l
            assert torch.equal(p.dx.view(torch.int16), dx), l
            assert torch.equal(p.dA, dA) and torch.equal(p.dB, dB), l
    rows = G.sample_rows(wl.T, 12, 3)
    for ps in layers:
        for p in ps:
            x, W, A, B, dy = (p.f64(k) for k in ("x", "W", "A", "B", "dy"))
            y_rows = oracle.lora_forward_rows(rows, x, W, A, B, p.s)
            dx_rows = oracle.lora_backward_dx_rows(rows, dy, W, A, B, p.s)
            dA, dB = oracle.lora_adapter_grads(dy, x, A, B, p.s)
            assert G.rel_fro(G.host_f64(p.y)[rows], y_rows) <= G.TOL_Y
            assert G.rel_fro(G.host_f64(p.dx)[rows], dx_rows) <= G.TOL_DX
            assert G.rel_fro(G.host_f64(p.dA), dA) <= G.TOL_GRAD
            assert G.rel_fro(G.host_f64(p.dB), dB) <= G.TOL_GRAD


def test_ckpt_argument_errors():
    wl = workloads.llama_sweep(256, 8)
    ps = build_layer(wl, seed=6)
    projs = [[p.proj() for p in ps]]
    need = lora.lora_stack_ckpt_workspace_size(projs)
    ws = G.workspace(need)
    with pytest.raises(lora.LoraError) as e:
        lora.lora_stack_ckpt(projs, ws, need - 256)
    assert e.value.code == lora.LORA_EWORKSPACE
    bad = [[lora.make_proj(p.shape, x=p.x, W=p.W, A=p.A, B=p.B, dy=None, y=p.y, dA=p.dA, dB=p.dB) for p in ps]]
    with pytest.raises(lora.LoraError) as e:
        lora.lora_stack_ckpt(bad, ws, need)
    assert e.value.code == lora.LORA_ENULL
    torch.cuda.synchronize()
    assert all(torch.isnan(p.y).all() for p in ps), "a rejected call must enqueue nothing"
