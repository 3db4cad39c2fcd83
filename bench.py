"""Benchmark of the LoRA-linear fwd+bwd hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference]

One step = forward then backward (lora_stack_step, LORA_FWD_BWD) of the seven
LoRA-adapted projections of a Llama-3.2-3B-shaped decoder layer (q, k, v, o,
gate, up, down; T = 2048 tokens, r = 16, alpha = 32), bf16 operands with fp32
accumulation, on seeded synthetic inputs.  Metric: tokens/s of fwd+bwd, and
the fraction of the GB300 dense-bf16 tensor peak it reaches.

Multi-GPU (torchrun, one process per GPU): every rank runs its own replica
on its own batch of T tokens (weak scaling, no collective on the data path);
value = total tokens of all ranks / max-over-ranks time.

--impl reference times the fp64 CPU oracle on this host's cores instead,
each step a bounded token sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2606_19528_gb300 import synth, workloads  # noqa: E402

METRIC = "LoRA-linear fwd+bwd tokens/s and % of GB300 dense-BF16 tensor peak (1 GPU)"
UNIT = "tokens/s"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20


GEMM_PROFILE = os.path.join(ROOT, "profiles", "fused_gemm_llama_layer_T2048_r16.md")
GEMM_SOURCES = ("paper_2606_19528_gb300/csrc/fused_gemm.cu", "paper_2606_19528_gb300/csrc/common.cuh")


def gemm_traffic(workload_name: str):
    """DRAM bytes per step of the two fused-GEMM launches from the committed ncu
    summary, or None when the workload differs or the kernel sources changed
    since the counters were taken."""
    import hashlib
    import re
    if workload_name != workloads.llama_layer_T2048().name:
        return None
    try:
        text = open(GEMM_PROFILE).read()
        h = hashlib.sha256()
        for f in GEMM_SOURCES:
            with open(os.path.join(ROOT, f), "rb") as fh:
                h.update(fh.read())
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_step:\s*(\d+)", text)
    sha = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    if not m or not sha or sha.group(1) != h.hexdigest():
        return None
    return int(m.group(1))


def load_peaks():
    try:
        with open(PEAKS_FILE) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


# ----------------------------------------------------------------------------- inputs

def gen_layer_bits(wl: workloads.Workload, seed: int = 0, T: int | None = None):
    """bf16 bits of every projection's inputs (x shared per input group)."""
    T = wl.T if T is None else T
    xs = {}
    out = []
    for i, p in enumerate(wl.projs):
        if p.group not in xs:
            xs[p.group] = synth.gen_x(seed, wl.cfg, p.group, 0, T, p.d_in)
        out.append({
            "x": xs[p.group], "group": p.group,
            "W": None if wl.q4 else synth.gen_W(seed, wl.cfg, i, 0, p.d_out, p.d_in),
            "A": synth.gen_A(seed, wl.cfg, i, 0, wl.rank, p.d_in),
            "B": synth.gen_B(seed, wl.cfg, i, 0, p.d_out, wl.rank, zero=wl.zero_B),
            "Wq": synth.gen_Wq(seed, wl.cfg, i, 0, p.d_out, p.d_in) if wl.q4 else None,
            "dy": synth.gen_dy(seed, wl.cfg, i, 0, T, p.d_out),
        })
    return out


def step_input_bytes(wl: workloads.Workload):
    """Bytes of one step's inputs: base weights (bf16, or 4-bit codes plus
    their (s, b) pairs), activations x (once per shared input) and dy."""
    T = wl.T
    w = sum(p.d_in * p.d_out * 2 if not wl.q4 else p.d_in * p.d_out // 2 + p.d_out * (p.d_in // 64) * 4
            for p in wl.projs)
    x = sum(T * p.d_in * 2 for g, p in {p.group: p for p in wl.projs}.items())
    dy = sum(T * p.d_out * 2 for p in wl.projs)
    return w * wl.layers, x * wl.layers, dy * wl.layers


def l2_note(wl: workloads.Workload) -> str:
    w, x, dy = step_input_bytes(wl)
    tot = w + x + dy
    mb = lambda b: f"{b / 1e6:.0f} MB"
    where = "also exceed" if tot > 129e6 else "fit in"
    return (f"256 MiB buffer written between timed steps (outside the step events); inputs of one step "
            f"({'4-bit ' if wl.q4 else ''}W {mb(w)} + x {mb(x)} + dy {mb(dy)} = {mb(tot)}) {where} the 129 MB L2")


def layer_config(wl: workloads.Workload, n_gpus: int) -> dict:
    """The workload's config key, the same in the GPU arm and the reference arm."""
    return {"workload": wl.name, "T": wl.T, "rank": wl.rank, "alpha": wl.alpha, "layers": wl.layers,
            "weights": "4-bit codes + (s, b) per 64-group" if wl.q4 else "bf16",
            "projections": [f"{p.name} {p.d_in}->{p.d_out}" for p in wl.projs],
            "step": step_desc(wl),
            "flops_per_step": wl.flops(),
            "l2": l2_note(wl),
            "parallelism": f"{n_gpus} independent replica(s), no collective"}


def gemm_flops(wl: workloads.Workload):
    """FLOPs the forward and backward fused-contraction launches of one step
    execute (every layer; the checkpointed schedule runs each forward twice)."""
    T, r = wl.T, wl.rank
    fwd = sum(2 * T * (p.d_in + r) * p.d_out for p in wl.projs) * wl.layers * (2 if wl.ckpt else 1)
    bwd = sum(2 * T * (p.d_out + r) * p.d_in for p in wl.projs) * wl.layers
    return float(fwd), float(bwd)


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id: str, period_ms: int = 100):
        self.cmd = ["nvidia-smi", "-i", gpu_id, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                    "-lms", str(period_ms)]
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "note": "nvidia-smi unavailable"}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, smax, power, reasons = [], [], [], set()
        for ln in self.lines:
            f = [c.strip() for c in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                smax.append(float(f[1]))
                power.append(float(f[2]))
            except ValueError:
                continue
            for name, v in zip(self.NAMES, f[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_max": max(power) if power else None}


# ----------------------------------------------------------------------------- CPU oracle timing

def oracle_sample(wl: workloads.Workload, tokens: int, seed: int = 0):
    """fp64 inputs of a `tokens`-token sample of the workload (outside timing);
    4-bit weights stay as codes and (s, b) pairs."""
    bits = gen_layer_bits(wl, seed, T=tokens)
    f = synth.bf16_bits_to_f64
    out = []
    for p in bits:
        e = {k: f(v) for k, v in p.items() if k not in ("group", "Wq", "W")}
        if p["Wq"] is not None:
            sb = f(p["Wq"][1])
            e["Wq"] = (p["Wq"][0], sb[..., 0], sb[..., 1])
        else:
            e["W"] = f(p["W"])
        out.append(e)
    return out


def time_oracle_step(sample, s: float):
    """One oracle fwd+bwd over the sample; 4-bit weights are dequantized
    (Algorithm 1) for the forward and again for the backward, inside the timing."""
    import oracle
    t0 = time.perf_counter()
    c0 = time.process_time()
    for p in sample:
        W = oracle.dequant_q4(*p["Wq"]) if "Wq" in p else p["W"]
        oracle.lora_forward(p["x"], W, p["A"], p["B"], s)
        W = oracle.dequant_q4(*p["Wq"]) if "Wq" in p else p["W"]
        oracle.lora_backward(p["dy"], p["x"], W, p["A"], p["B"], s)
    return time.perf_counter() - t0, time.process_time() - c0


def cpu_baseline(wl: workloads.Workload, budget_s: float = 15.0):
    """The oracle as it stands on this host's cores, over a token sample sized
    to about `budget_s` seconds of work; tokens/s of the full fwd+bwd."""
    probe_T = 64
    sample = oracle_sample(wl, probe_T)
    time_oracle_step(sample, wl.scale)  # warm BLAS threads
    wall, _ = time_oracle_step(sample, wl.scale)
    T = int(min(wl.T, max(64, probe_T * budget_s / max(wall, 1e-3) / 2)))
    T = max(8, T // 8 * 8)
    sample = oracle_sample(wl, T)
    walls, cpus = [], []
    t_start = time.perf_counter()
    while time.perf_counter() - t_start < budget_s / 2 or not walls:
        w, c = time_oracle_step(sample, wl.scale)
        walls.append(w)
        cpus.append(c)
    wall = sum(walls) / len(walls)
    cores_used = max(1, round(sum(cpus) / sum(walls)))
    return {"value": T / wall, "unit": UNIT, "cores": cores_used, "kind": "oracle",
            "host_cpus": os.cpu_count(),
            "sample": f"fp64 oracle (numpy BLAS) fwd+bwd of all {len(wl.projs)} projections on {T} of the "
                      f"workload's {wl.T} tokens, {len(walls)} repetitions, mean {wall:.3f} s each"}


def run_reference(args, wl):
    """--impl reference: the oracle timed as the reference arm."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    W, K = args.warmup, args.steps
    probe = oracle_sample(wl, 32)
    time_oracle_step(probe, wl.scale)
    w32, _ = time_oracle_step(probe, wl.scale)
    # tokens per step so that warmup + steps fit in about 90 s
    per_step_budget = 90.0 / max(1, W + K)
    T = int(32 * per_step_budget / max(w32, 1e-4))
    T = max(8, min(wl.T, T // 8 * 8))
    sample = oracle_sample(wl, T)
    for _ in range(W):
        time_oracle_step(sample, wl.scale)
    walls, cpus = [], []
    for _ in range(K):
        w, c = time_oracle_step(sample, wl.scale)
        walls.append(w)
        cpus.append(c)
    total = sum(walls)
    value = T * K / total
    cores = max(1, round(sum(cpus) / total))
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": K, "warmup": W, "ms_per_step": 1e3 * total / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": layer_config(wl, args.gpus),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "host_cpus": os.cpu_count(), "sample_tokens_per_step": T,
                         "sample": f"{T} of {wl.T} tokens per step, all {len(wl.projs)} projections fwd+bwd"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- distributed helpers

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if world <= 1:
        return None, 0, 1
    import torch.distributed as dist
    backend = "nccl" if os.environ.get("BENCH_DIST_BACKEND", "nccl") == "nccl" else "gloo"
    dist.init_process_group(backend=backend)
    return dist, dist.get_rank(), dist.get_world_size()


def max_over_ranks(dist, value: float, device=None) -> float:
    """Max of a host float over ranks (timing aggregation only, not the data path)."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist, device=None):
    if dist is not None:
        if device is not None:
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


def sustained_pass(torch, lora, step, stream, step_ms, gpu_id, seconds):
    """Steps back to back (no L2 flush; the inputs exceed the L2) for about
    `seconds`, twice: first with events at the two ends only (whole steps),
    then with the library's events around the fused-GEMM launches.  Returns
    their per-step times and the clock record of the first pass."""
    n = max(10, int(seconds * 1e3 / max(step_ms, 1e-3)))
    sampler = ClockSampler(gpu_id) if gpu_id else None
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
        time.sleep(0.3)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(n):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    clk = sampler.stop() if sampler else None
    whole_ms = e0.elapsed_time(e1) / n
    lora.lora_profile_begin((lora.LORA_KERNEL_GEMM_FWD, lora.LORA_KERNEL_GEMM_BWD))
    for _ in range(n):
        step()
    torch.cuda.synchronize()
    kern_ms, _ = lora.lora_profile_end()
    return {"steps": n, "seconds": whole_ms * n / 1e3, "ms_per_step": whole_ms,
            "gemm_ms_per_step": (kern_ms["gemm_fwd"] + kern_ms["gemm_bwd"]) / n, "clocks": clk,
            "note": "steps back to back without the L2 flush for the stated seconds (events at the two ends "
                    "only), then as many steps again with events around the fused-GEMM launches; fractions "
                    "against the measured sustained bf16 peak"}


KERNEL_PASS_NOTE = ("launch durations from CUDA events around each launch of this kernel over a second pass of "
                    "the same K steps, run right after the timed region; the timed region itself records "
                    "events around whole steps only, because an event between two launches stops "
                    "programmatic dependent launch there")


def timed_passes(torch, lora, step, K, stream, flush=None, kinds=(0, 1)):
    """The timed region, then the kernel pass.

    Timed region: K steps with events around each step only (L2 flushed
    between steps when `flush` is given).  Kernel pass: the same K steps
    with the library's events around every launch of `kinds`.  Returns
    (per-step ms of the timed region, {kind: device ms per step} of the
    kernel pass, library launches inside the timed region)."""
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    torch.cuda.synchronize()
    launches0 = lora.lora_launch_count()
    for i in range(K):
        if flush is not None:
            flush.zero_()
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    launches = lora.lora_launch_count() - launches0
    step_ms = [a.elapsed_time(b) for a, b in ev]
    lora.lora_profile_begin(kinds)
    for _ in range(K):
        if flush is not None:
            flush.zero_()
        step()
    torch.cuda.synchronize()
    kern_ms, _ = lora.lora_profile_end()
    return step_ms, {k: v / K for k, v in kern_ms.items()}, launches


# ----------------------------------------------------------------------------- GPU arm

class LayerOnDevice:
    def __init__(self, wl, bits, torch, lora):
        self.wl = wl
        self.torch = torch
        dev = torch.device("cuda")

        def d(b):
            return torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(dev).view(torch.bfloat16)

        T, r = wl.T, wl.rank
        xs = {}
        self.p = []
        for pb, pr in zip(bits, wl.projs):
            if pr.group not in xs:
                xs[pr.group] = d(pb["x"])
            wq = None
            if pb["Wq"] is not None:
                codes = torch.from_numpy(pb["Wq"][0]).to(dev)
                params = d(pb["Wq"][1])
                wq = (codes, params, lora.make_q4(codes, params))
            e = {"x": xs[pr.group], "W": None if wq else d(pb["W"]), "Wq": wq,
                 "A": d(pb["A"]), "B": d(pb["B"]), "dy": d(pb["dy"]),
                 "y": torch.empty(T, pr.d_out, dtype=torch.bfloat16, device=dev),
                 "su": torch.empty(T, r, dtype=torch.bfloat16, device=dev),
                 "dx": torch.empty(T, pr.d_in, dtype=torch.bfloat16, device=dev),
                 "dA": torch.empty(r, pr.d_in, dtype=torch.float32, device=dev),
                 "dB": torch.empty(pr.d_out, r, dtype=torch.float32, device=dev)}
            self.p.append(e)
        self.xs = xs
        self.projs = [lora.make_proj(lora.make_shape(T, pr.d_in, pr.d_out, r, wl.scale), x=e["x"], W=e["W"],
                                     A=e["A"], B=e["B"], dy=e["dy"], y=e["y"], su=e["su"], dx=e["dx"], dA=e["dA"],
                                     dB=e["dB"], Wq=e["Wq"][2] if e["Wq"] else None)
                      for e, pr in zip(self.p, wl.projs)]
        n = lora.lora_stack_workspace_size(self.projs, lora.LORA_FWD_BWD)
        self.ws = torch.empty(max(n, 256), dtype=torch.uint8, device=dev)

    def second_input_set(self, lora):
        """A second set of x and dy buffers with descriptors that share every
        other tensor (weights, outputs, workspace): the double buffer of a
        loader that copies the next step's inputs while this step runs."""
        torch, T, r = self.torch, self.wl.T, self.wl.rank
        xs2 = {g: torch.empty_like(t) for g, t in self.xs.items()}
        dys2 = [torch.empty_like(e["dy"]) for e in self.p]
        projs2 = [lora.make_proj(lora.make_shape(T, pr.d_in, pr.d_out, r, self.wl.scale), x=xs2[pr.group],
                                 W=e["W"], A=e["A"], B=e["B"], dy=dy, y=e["y"], su=e["su"], dx=e["dx"],
                                 dA=e["dA"], dB=e["dB"], Wq=e["Wq"][2] if e["Wq"] else None)
                  for e, pr, dy in zip(self.p, self.wl.projs, dys2)]
        return xs2, dys2, projs2

    def step(self, lora, stream, projs=None):
        lora.lora_stack_step(self.projs if projs is None else projs, lora.LORA_FWD_BWD, self.ws, self.ws.numel(),
                             stream)


class StackOnDevice:
    """`wl.layers` layers of the workload's projections, each with its own
    buffers (filled with the first layer's synthetic values), run forward of
    every layer then backward of every layer in reverse, or with the
    checkpointed schedule (Algorithm 2) when `wl.ckpt`."""

    def __init__(self, wl, bits, torch, lora):
        self.wl = wl
        first = LayerOnDevice(wl, bits, torch, lora)
        self.layers = [first]
        for _ in range(wl.layers - 1):
            L = LayerOnDevice.__new__(LayerOnDevice)
            L.wl, L.torch = wl, torch
            L.xs = {g: t.clone() for g, t in first.xs.items()}
            L.p = []
            for e, pr in zip(first.p, wl.projs):
                c = {k: (v.clone() if hasattr(v, "clone") else v) for k, v in e.items() if k != "x"}
                c["x"] = L.xs[pr.group]
                L.p.append(c)
            L.projs = [lora.make_proj(lora.make_shape(wl.T, pr.d_in, pr.d_out, wl.rank, wl.scale), x=e["x"],
                                      W=e["W"], A=e["A"], B=e["B"], dy=e["dy"], y=e["y"], su=e["su"], dx=e["dx"],
                                      dA=e["dA"], dB=e["dB"], Wq=None) for e, pr in zip(L.p, wl.projs)]
            self.layers.append(L)
        self.p = [e for L in self.layers for e in L.p]
        self.lora = lora
        layer_projs = [L.projs for L in self.layers]
        if wl.ckpt:
            n = lora.lora_stack_ckpt_workspace_size(layer_projs)
        else:
            n = max(max(lora.lora_stack_workspace_size(L.projs, m) for m in (lora.LORA_FWD, lora.LORA_BWD))
                    for L in self.layers)
        self.ws = torch.empty(max(n, 256), dtype=torch.uint8, device="cuda")

    def step(self, lora, stream, projs=None):
        if self.wl.ckpt:
            lora.lora_stack_ckpt([L.projs for L in self.layers], self.ws, self.ws.numel(), stream)
            return
        for L in self.layers:
            lora.lora_stack_step(L.projs, lora.LORA_FWD, self.ws, self.ws.numel(), stream)
        for L in reversed(self.layers):
            lora.lora_stack_step(L.projs, lora.LORA_BWD, self.ws, self.ws.numel(), stream)


def step_desc(wl) -> str:
    n = len(wl.projs)
    if wl.layers == 1:
        return f"lora_stack_step(LORA_FWD_BWD): {n} forwards then {n} backwards"
    if wl.ckpt:
        return (f"lora_stack_ckpt over {wl.layers} layers of {n} projections: every forward saving nothing, "
                "then per layer from the last a re-forward and the backward (Algorithm 2)")
    return f"{wl.layers} layers of {n} projections: every forward (saving su), then every backward in reverse"


# ----------------------------------------------------------------------------- LM-head cross entropy

_CE_STATIC = {}


def ce_inputs(wl, seed: int = 0, T: int | None = None):
    """Seeded inputs of the LM-head workload (targets, mask and top-k table
    with the locality described in synth); E and the table are drawn once."""
    T = wl.T if T is None else T
    key = (wl.name, seed)
    if key not in _CE_STATIC:
        E = synth.gen_E(seed, wl.cfg, wl.vocab, wl.hidden)
        tab = synth.gen_topk_table(seed, wl.cfg, wl.vocab, wl.topk, wl.cluster) if wl.topk else None
        _CE_STATIC[key] = (E, tab)
    E, tab = _CE_STATIC[key]
    h = synth.gen_h(seed, wl.cfg, T, wl.hidden)
    y = synth.gen_targets(seed, wl.cfg, T, wl.vocab, wl.cluster)
    m = synth.gen_mask(T, wl.trainable)
    return h, E, y, m, tab


def run_gpu_ce(args, wl):
    """The LM-head node: reduced-vocabulary cross entropy with logits masking."""
    import torch

    from paper_2606_19528_gb300 import lora

    dist, rank, world = dist_setup()
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    lora.library()
    peaks, peaks_src = load_peaks()
    h, E, y, m, tab = ce_inputs(wl, seed=rank)
    dev = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(device).view(torch.bfloat16)
    d_h, d_E = dev(h), dev(E)
    d_y, d_m = torch.from_numpy(y).to(device), torch.from_numpy(m).to(device)
    d_tab = torch.from_numpy(tab).to(device) if tab is not None else None
    loss = torch.empty(1, device=device)
    token_loss = torch.empty(wl.T, device=device)
    dh = torch.empty(wl.T, wl.hidden, dtype=torch.bfloat16, device=device)
    args_ce = lora.make_ce_args(wl.T, wl.hidden, wl.vocab, d_h, d_E, d_y, loss, mask=d_m, topk=d_tab,
                                ld_topk=wl.topk, k=wl.topk, token_loss=token_loss, dh=dh)
    ws = torch.empty(lora.lora_ce_workspace_size(args_ce), dtype=torch.uint8, device=device)
    stream = torch.cuda.current_stream()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

    def step():
        return lora.lora_ce_fwd_bwd(args_ce, ws, ws.numel(), stream)

    W, K = max(3, args.warmup), args.steps
    for _ in range(W):
        nT, nJ = step()
    torch.cuda.synchronize()
    props = torch.cuda.get_device_properties(device)
    gpu_id = str(getattr(props, "uuid", local))
    if gpu_id and not gpu_id.startswith("GPU-") and len(gpu_id) == 36:
        gpu_id = "GPU-" + gpu_id
    clocks = ClockSampler(gpu_id) if rank == 0 else None
    barrier(dist, device)
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
        time.sleep(0.3)
    steps_ms, kern_ms, launches = timed_passes(torch, lora, step, K, stream, flush,
                                               (lora.LORA_KERNEL_GEMM_FWD, lora.LORA_KERNEL_GEMM_BWD))
    barrier(dist, device)
    clk = clocks.stop() if clocks else None
    step_ms = max_over_ranks(dist, sum(steps_ms) / K, device)

    # end to end: h, targets and mask from pinned host memory, loss back, every step
    h_h = torch.from_numpy(np.ascontiguousarray(h).view(np.int16)).pin_memory()
    h_y, h_m = torch.from_numpy(y).pin_memory(), torch.from_numpy(m).pin_memory()
    h_loss = torch.empty(1).pin_memory()
    Ke = max(10, min(K, 100))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(Ke):
        d_h.view(torch.int16).copy_(h_h, non_blocking=True)
        d_y.copy_(h_y, non_blocking=True)
        d_m.copy_(h_m, non_blocking=True)
        step()
        h_loss.copy_(loss, non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(dist, e0.elapsed_time(e1) / Ke, device)
    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0
    gemm_ms = kern_ms["gemm_fwd"] + kern_ms["gemm_bwd"]
    flops = 4.0 * nT * nJ * wl.hidden  # logits and dh contractions
    sustained = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    burst = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    gemm_tf = flops / (gemm_ms / 1e3) / 1e12 if gemm_ms > 0 else None
    line = {
        "metric": METRIC, "value": world * wl.T / (step_ms / 1e3), "unit": UNIT, "n_gpus": world,
        "steps": K, "warmup": W, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": wl.name, "T": wl.T, "vocab": wl.vocab, "hidden": wl.hidden, "topk": wl.topk,
                   "trainable_fraction": wl.trainable, "trainable_positions": nT, "reduced_vocab": nJ,
                   "step": "lora_ce_fwd_bwd: index pass, logits of trainable positions over J, softmax CE, dh",
                   "l2": "256 MiB buffer written between timed steps (outside the step events)",
                   "parallelism": f"{world} independent replica(s), no collective"},
        "tflops": flops / (step_ms / 1e3) / 1e12,
        "roofline": {"kernel": "fused_lora_gemm (logits and dh contractions)", "bound": "tensor",
                     "achieved": gemm_tf, "peak": burst, "unit": "TFLOP/s",
                     "frac": gemm_tf / burst if gemm_tf else None, "traffic": None,
                     "peak_kind": f"bf16 burst, of {peaks_src} (short timed region)",
                     "frac_of_sustained": gemm_tf / sustained if gemm_tf else None,
                     "flops_per_step": flops, "ms_per_step": gemm_ms,
                     "timing": KERNEL_PASS_NOTE},
        "gpu_launches": launches,
        "clocks": clk,
        "status": lora.lora_strerror(lora.lora_read_status()),
        "e2e": {"value": world * wl.T / (e2e_ms / 1e3), "unit": UNIT, "ms_per_step": e2e_ms, "steps": Ke,
                "h2d_bytes_per_step": h_h.numel() * 2 + h_y.numel() * 4 + h_m.numel(),
                "d2h_bytes_per_step": 4},
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline_ce(wl, budget_s=args.cpu_budget)
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def time_oracle_ce(wl, T: int):
    import oracle
    h, E, y, m, tab = ce_inputs(wl, T=T)
    hf, Ef = synth.bf16_bits_to_f64(h), synth.bf16_bits_to_f64(E)
    mb = m.astype(bool)
    t0, c0 = time.perf_counter(), time.process_time()
    J = np.arange(wl.vocab) if tab is None else oracle.reduced_vocab(y, mb, tab, wl.topk)
    oracle.ce_forward_backward(hf, Ef, y, mb, J)
    return time.perf_counter() - t0, time.process_time() - c0


def cpu_baseline_ce(wl, budget_s: float = 15.0):
    """The oracle on the host cores over the first positions of the sequence."""
    T = 64
    w, _ = time_oracle_ce(wl, T)
    T = int(min(wl.T, max(64, T * budget_s / max(w, 1e-3) / 2)))
    w, c = time_oracle_ce(wl, T)
    return {"value": T / w, "unit": UNIT, "cores": max(1, round(c / w)), "kind": "oracle",
            "host_cpus": os.cpu_count(),
            "sample": f"fp64 oracle on the first {T} of {wl.T} positions (same trainable fraction), one run, "
                      f"{w:.2f} s"}


def run_gpu_topk(args, wl):
    """The top-k similarity table of the embedding: one step builds the whole table."""
    import torch

    from paper_2606_19528_gb300 import lora

    torch.cuda.set_device(0)
    device = torch.device("cuda", 0)
    lora.library()
    peaks, peaks_src = load_peaks()
    V, d, k = wl.vocab, wl.hidden, wl.topk
    E = torch.from_numpy(np.ascontiguousarray(synth.gen_E(0, wl.cfg, V, d)).view(np.int16)).to(device)
    table = torch.empty(V, k, dtype=torch.int32, device=device)
    ws = torch.empty(lora.lora_topk_workspace_size(V, d, k), dtype=torch.uint8, device=device)
    stream = torch.cuda.current_stream()

    def step():
        lora.lora_topk_table(E, V, d, k, table, ws, ws.numel(), stream)

    W, K = max(1, min(args.warmup, 2)), max(1, min(args.steps, 5))
    for _ in range(W):
        step()
    torch.cuda.synchronize()
    props = torch.cuda.get_device_properties(device)
    gpu_id = str(getattr(props, "uuid", 0))
    if gpu_id and not gpu_id.startswith("GPU-") and len(gpu_id) == 36:
        gpu_id = "GPU-" + gpu_id
    clocks = ClockSampler(gpu_id)
    clocks.start()
    time.sleep(0.3)
    steps_ms, kern_ms, launches = timed_passes(torch, lora, step, K, stream, None, (lora.LORA_KERNEL_GEMM_FWD,))
    clk = clocks.stop()
    step_ms = sum(steps_ms) / K
    gemm_ms = kern_ms["gemm_fwd"]
    flops = 2.0 * V * V * d
    if V >= 32768:
        # the contractions performed: each row against 8192 sample tokens (thresholds), and the upper
        # triangle of C = E~ E~^T in 512-row blocks (block I against tokens from 512 I on)
        done_flops = 2.0 * V * 8192 * d + sum(2.0 * min(512, V - a0) * (V - a0) * d for a0 in range(0, V, 512))
    else:
        done_flops = flops
    sustained = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    burst = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    gemm_tf = done_flops / (gemm_ms / 1e3) / 1e12
    line = {
        "metric": "top-k similarity table rows/s", "value": V / (step_ms / 1e3), "unit": "rows/s", "n_gpus": 1,
        "steps": K, "warmup": W, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "strong",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": wl.name, "vocab": V, "hidden": d, "k": k,
                   "step": "lora_topk_table: normalise; per-row thresholds from a contraction against 8192 "
                           "evenly spread tokens; the upper triangle of the similarities in tcgen05 contractions "
                           "whose epilogue keeps each value at or above either of its rows' thresholds; then a "
                           "per-row sort",
                   "tflops_counts": "contractions performed (sample + upper triangle), not 2 V^2 d"},
        "tflops": done_flops / (step_ms / 1e3) / 1e12,
        "roofline": {"kernel": "fused_lora_gemm (sample and similarity contractions)", "bound": "tensor",
                     "achieved": gemm_tf, "peak": sustained, "unit": "TFLOP/s", "frac": gemm_tf / sustained,
                     "traffic": None,
                     "peak_kind": f"bf16 sustained, of {peaks_src} (each step runs {step_ms / 1e3:.3f} s)",
                     "frac_of_burst": gemm_tf / burst, "flops_per_step": done_flops, "ms_per_step": gemm_ms,
                     "timing": KERNEL_PASS_NOTE},
        "gpu_launches": launches, "clocks": clk, "status": lora.lora_strerror(lora.lora_read_status()),
        "e2e": None,
    }
    print(json.dumps(line), flush=True)
    return 0


def run_reference_ce(args, wl):
    """--impl reference for the LM-head workload: the oracle on a bounded sample of positions."""
    if int(os.environ.get("RANK", "0")) != 0:
        return 0
    W, K = args.warmup, args.steps
    w64, _ = time_oracle_ce(wl, 64)
    T = int(min(wl.T, max(64, 64 * (90.0 / max(1, W + K)) / max(w64, 1e-3))))
    for _ in range(W):
        time_oracle_ce(wl, T)
    walls, cpus = [], []
    for _ in range(K):
        w, c = time_oracle_ce(wl, T)
        walls.append(w)
        cpus.append(c)
    total = sum(walls)
    value = T * K / total
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": K,
            "warmup": W, "ms_per_step": 1e3 * total / K, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": wl.name, "T": wl.T, "vocab": wl.vocab, "hidden": wl.hidden, "topk": wl.topk,
                       "sample_positions_per_step": T},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": max(1, round(sum(cpus) / total)),
                             "kind": "oracle", "host_cpus": os.cpu_count(),
                             "sample": f"first {T} of {wl.T} positions per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_gpu(args, wl):
    import torch

    from paper_2606_19528_gb300 import lora

    dist, rank, world = dist_setup()
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    lora.library()
    peaks, peaks_src = load_peaks()

    bits = gen_layer_bits(wl, seed=rank)
    if wl.layers > 1:
        if wl.q4:
            raise SystemExit("stack workloads use bf16 weights")
        L = StackOnDevice(wl, bits, torch, lora)
        args.no_e2e = True  # the end-to-end copies are defined for the single-layer workloads
    else:
        L = LayerOnDevice(wl, bits, torch, lora)
    stream = torch.cuda.current_stream()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=device)

    W, K = max(3, args.warmup), args.steps
    for _ in range(W):
        L.step(lora, stream)
    # a short profiled pass so that the event pool exists before the timed region
    lora.lora_profile_begin()
    L.step(lora, stream)
    lora.lora_profile_end()
    torch.cuda.synchronize()
    assert lora.lora_read_status() == lora.LORA_OK

    props = torch.cuda.get_device_properties(device)
    gpu_id = str(getattr(props, "uuid", local))
    if gpu_id and not gpu_id.startswith("GPU-") and len(gpu_id) == 36:
        gpu_id = "GPU-" + gpu_id

    # ---------------- timed region: device-resident inputs, L2 flushed between steps;
    # then the kernel pass (events around the fused-GEMM launches)
    clocks = ClockSampler(gpu_id) if rank == 0 else None
    barrier(dist, device)
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
        time.sleep(0.3)
    steps_ms, kern_ms, launches = timed_passes(torch, lora, lambda: L.step(lora, stream), K, stream, flush,
                                               (lora.LORA_KERNEL_GEMM_FWD, lora.LORA_KERNEL_GEMM_BWD))
    barrier(dist, device)
    clk = clocks.stop() if clocks else None
    status = lora.lora_read_status()
    step_ms_local = sum(steps_ms) / K
    step_ms = max_over_ranks(dist, step_ms_local, device)

    # ---------------- sustained: back-to-back steps for seconds, with their own clock record
    sustained_rec = None
    if not args.no_sustained:
        sustained_rec = sustained_pass(torch, lora, lambda: L.step(lora, stream), stream, step_ms_local,
                                       gpu_id if rank == 0 else None, args.sustained_s)

    # ---------------- per-kind breakdown: a separate pass with events around every launch group
    Kb = max(10, min(K, 100))
    lora.lora_profile_begin()
    for i in range(Kb):
        flush.zero_()
        L.step(lora, stream)
    torch.cuda.synchronize()
    brk_ms, brk_launches = lora.lora_profile_end()

    # ---------------- comparison (never the metric): the same forward and backward written as a
    # composition of torch.matmul calls (cuBLAS, bf16 in, fp32 accumulate), same buffers, same L2 flush
    composition = None
    if wl.layers == 1 and not wl.q4 and rank == 0:
        s = wl.scale

        def torch_step():
            for e in L.p:
                x, W, A, B, dy = e["x"], e["W"], e["A"], e["B"], e["dy"]
                u = x @ A.t()
                su = u * s
                e["y"].copy_(x @ W.t() + su @ B.t())
                sv = (dy @ B) * s
                e["dx"].copy_(dy @ W + sv @ A)
                e["dB"].copy_((dy.t() @ su).float())
                e["dA"].copy_((sv.t() @ x).float())

        for _ in range(3):
            torch_step()
        torch.cuda.synchronize()
        cev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(20)]
        for a, b in cev:
            flush.zero_()
            a.record(stream)
            torch_step()
            b.record(stream)
        torch.cuda.synchronize()
        comp_ms = sum(a.elapsed_time(b) for a, b in cev) / len(cev)
        composition = {"ms_per_step": comp_ms, "value": wl.T / (comp_ms / 1e3), "unit": UNIT,
                       "library_speedup": comp_ms / step_ms,
                       "note": "torch.matmul (cuBLAS) bf16 composition of the same forward and backward over the "
                               "same device buffers (u = x A^T, y = x W^T + s u B^T, v = dy B, dx = dy W + s v A, "
                               "dB = s dy^T u, dA = s v^T x), L2 flushed between steps; a comparison, not the "
                               "measured path"}
        L.step(lora, stream)  # leave the library's outputs in the buffers
        torch.cuda.synchronize()

    # ---------------- end-to-end: host inputs (pinned) -> device -> step -> gradients back to host
    e2e = None
    if not args.no_e2e:
        h_x = {g: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).pin_memory()
               for g, b in ((pb["group"], pb["x"]) for pb in bits)}
        h_dy = [torch.from_numpy(np.ascontiguousarray(pb["dy"]).view(np.int16)).pin_memory() for pb in bits]
        h_dA = [torch.empty(e["dA"].shape, dtype=torch.float32).pin_memory() for e in L.p]
        h_dB = [torch.empty(e["dB"].shape, dtype=torch.float32).pin_memory() for e in L.p]
        h2d_bytes = sum(t.numel() * 2 for t in h_x.values()) + sum(t.numel() * 2 for t in h_dy)
        d2h_bytes = sum(t.numel() * 4 for t in h_dA) + sum(t.numel() * 4 for t in h_dB)

        def e2e_step():
            for g, t in h_x.items():
                L.xs[g].view(torch.int16).copy_(t, non_blocking=True)
            for e, t in zip(L.p, h_dy):
                e["dy"].view(torch.int16).copy_(t, non_blocking=True)
            L.step(lora, stream)
            for e, a, b in zip(L.p, h_dA, h_dB):
                a.copy_(e["dA"], non_blocking=True)
                b.copy_(e["dB"], non_blocking=True)

        Ke = max(10, min(K, 200))
        for _ in range(3):
            e2e_step()
        torch.cuda.synchronize()
        barrier(dist, device)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(Ke):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        serial_ms = max_over_ranks(dist, e0.elapsed_time(e1) / Ke, device)

        # pipelined: a copy stream fills the other input set while this step
        # computes; the gradients go back on the compute stream (they are
        # overwritten by the next step)
        xs2, dys2, projs2 = L.second_input_set(lora)
        sets = [(L.xs, [e["dy"] for e in L.p], L.projs), (xs2, dys2, projs2)]
        copy = torch.cuda.Stream(device=device)
        ev_in = [torch.cuda.Event() for _ in range(2)]
        ev_free = [torch.cuda.Event() for _ in range(2)]

        def h2d(k):
            xs_k, dys_k, _ = sets[k]
            copy.wait_event(ev_free[k])
            with torch.cuda.stream(copy):
                for g, t in h_x.items():
                    xs_k[g].view(torch.int16).copy_(t, non_blocking=True)
                for d_, t in zip(dys_k, h_dy):
                    d_.view(torch.int16).copy_(t, non_blocking=True)
            ev_in[k].record(copy)

        def pipelined(n):
            for k in range(2):
                ev_free[k].record(stream)
            h2d(0)
            for i in range(n):
                k = i % 2
                if i + 1 < n:
                    h2d(1 - k)
                stream.wait_event(ev_in[k])
                L.step(lora, stream, sets[k][2])
                ev_free[k].record(stream)
                for e, a, b in zip(L.p, h_dA, h_dB):
                    a.copy_(e["dA"], non_blocking=True)
                    b.copy_(e["dB"], non_blocking=True)

        pipelined(3)
        torch.cuda.synchronize()
        barrier(dist, device)
        e0.record(stream)
        pipelined(Ke)
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(dist, e0.elapsed_time(e1) / Ke, device)
        # the same host-to-device copies alone: the link rate the pipelined steps are bounded by
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        c0.record(copy)
        for _ in range(10):
            with torch.cuda.stream(copy):
                for g, t in h_x.items():
                    xs2[g].view(torch.int16).copy_(t, non_blocking=True)
                for d_, t in zip(dys2, h_dy):
                    d_.view(torch.int16).copy_(t, non_blocking=True)
        c1.record(copy)
        torch.cuda.synchronize()
        copy_ms = c0.elapsed_time(c1) / 10
        e2e = {"value": world * wl.T / (e2e_ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d_bytes,
               "d2h_bytes_per_step": d2h_bytes, "ms_per_step": e2e_ms, "steps": Ke,
               "serial_ms_per_step": serial_ms, "h2d_only_ms_per_step": copy_ms,
               "h2d_gbs": h2d_bytes / (copy_ms / 1e3) / 1e9,
               "note": "every step copies its x and dy from pinned host memory and its dA, dB back to pinned "
                       "host memory; the copy of step i+1's inputs (copy stream, second input buffer) "
                       "overlaps step i; serial_ms_per_step: copies and step on one stream; h2d_only: the "
                       "input copies alone, the host link rate that bounds the pipelined steps"}

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0

    flops = wl.flops()
    tflops = flops / (step_ms / 1e3) / 1e12
    f_fwd, f_bwd = gemm_flops(wl)
    gemm_ms = kern_ms["gemm_fwd"] + kern_ms["gemm_bwd"]
    gemm_tflops = (f_fwd + f_bwd) / (gemm_ms / 1e3) / 1e12
    sustained = peaks.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"])
    burst = peaks.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"])
    if sustained_rec is not None:
        sr = sustained_rec
        sr["tflops"] = flops / (sr["ms_per_step"] / 1e3) / 1e12
        sr["frac_of_sustained"] = sr["tflops"] / sustained
        sr["gemm_tflops"] = (f_fwd + f_bwd) / (sr["gemm_ms_per_step"] / 1e3) / 1e12
        sr["gemm_frac_of_sustained"] = sr["gemm_tflops"] / sustained
        sr["tokens_per_s"] = world * wl.T / (sr["ms_per_step"] / 1e3)
    per_kernel = {k: {"ms_per_step": brk_ms[k] / Kb, "launches_per_step": brk_launches[k] / Kb,
                      "share": brk_ms[k] / max(1e-9, sum(brk_ms.values()))} for k in brk_ms}
    per_kernel["note"] = (f"separate pass of {Kb} steps with events around every launch group "
                          "(which also stops programmatic dependent launch between groups)")
    line = {
        "metric": METRIC, "value": world * wl.T / (step_ms / 1e3), "unit": UNIT, "n_gpus": world,
        "steps": K, "warmup": W, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": layer_config(wl, world),
        "tflops": tflops,
        "pct_of_bf16_peak": {"sustained": tflops / sustained, "burst": tflops / burst,
                             "peak_tflops_sustained": sustained, "peak_tflops_burst": burst,
                             "source": peaks_src},
        "roofline": {"kernel": "fused_lora_gemm (fwd and bwd launches)", "bound": "tensor",
                     "achieved": gemm_tflops, "peak": burst, "unit": "TFLOP/s",
                     "frac": gemm_tflops / burst, "traffic": gemm_traffic(wl.name),
                     "traffic_unit": "bytes per step (forward + backward launch), ncu dram__bytes_read+write",
                     "peak_kind": f"bf16 burst, of {peaks_src} (the timed region lasts "
                                  f"{K * step_ms / 1e3:.3f} s; the seconds-long pass is under 'sustained')",
                     "frac_of_sustained": gemm_tflops / sustained,
                     "flops_per_step": f_fwd + f_bwd, "ms_per_step": gemm_ms,
                     "timing": KERNEL_PASS_NOTE},
        "sustained": sustained_rec,
        "kernels": per_kernel,
        "gpu_launches": launches,
        "clocks": clk,
        "status": lora.lora_strerror(status),
        "e2e": e2e,
        "cublas_composition": composition,
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, budget_s=args.cpu_budget)
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=("gb300", "reference"), default="gb300")
    ap.add_argument("--workload", default="llama_layer", choices=sorted(workloads.BY_NAME))
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-sustained", action="store_true", help="skip the seconds-long back-to-back pass")
    ap.add_argument("--sustained-s", type=float, default=2.5)
    ap.add_argument("--sweep", action="store_true",
                    help="the Llama layer over T in {256, 1024, 4096, 16384} x r in {4 .. 128} (one JSON line per "
                         "point; device-timed steps only)")
    args = ap.parse_args(argv)
    if args.sweep:
        args.no_e2e = args.no_cpu_baseline = args.no_sustained = True
        rc = 0
        for T in workloads.SWEEP_TOKENS:
            for r in workloads.SWEEP_RANKS:
                rc |= run_gpu(args, workloads.llama_sweep(T, r))
        return rc
    wl = workloads.BY_NAME[args.workload]()
    if wl.kind == "topk":
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable": "the top-k table workload has no CPU arm: "
                              "exact similarities of 128256 x 128256 pairs take hours on the host"}))
            return 0
        return run_gpu_topk(args, wl)
    if wl.kind == "ce":
        return run_reference_ce(args, wl) if args.impl == "reference" else run_gpu_ce(args, wl)
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_gpu(args, wl)


if __name__ == "__main__":
    sys.exit(main())
