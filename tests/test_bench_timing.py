"""CPU tests of bench.py's timing protocol with fake CUDA events and a fake
library: the timed region brackets whole steps only (no per-launch events,
which would stop programmatic dependent launch between the step's kernels),
flushes the L2 before every timed step, counts the library's launches of the
timed steps alone, and the launch durations of the roofline kernel come from
a second pass of the same number of steps with profiling on."""
import types

import bench


class FakeEvent:
    clock = [0.0]

    def __init__(self, enable_timing=False):
        self.t = None

    def record(self, stream=None):
        self.t = FakeEvent.clock[0]

    def elapsed_time(self, other):
        return other.t - self.t


class FakeLib:
    def __init__(self, log):
        self.log = log
        self.launches = 0
        self.profiling = False

    def lora_launch_count(self):
        return self.launches

    def lora_profile_begin(self, kinds=None):
        self.log.append(("profile_begin", tuple(kinds) if kinds else None))
        self.profiling = True

    def lora_profile_end(self):
        self.log.append(("profile_end",))
        self.profiling = False
        return {"gemm_fwd": 6.0, "gemm_bwd": 4.0}, {"gemm_fwd": 3, "gemm_bwd": 3}


def _fake_torch(log):
    cuda = types.SimpleNamespace(Event=FakeEvent, synchronize=lambda: log.append(("sync",)))
    return types.SimpleNamespace(cuda=cuda)


def test_timed_region_has_no_profiling_and_kernel_pass_does():
    log = []
    lib = FakeLib(log)
    flush = types.SimpleNamespace(zero_=lambda: log.append(("flush",)))

    def step():
        log.append(("step", lib.profiling))
        lib.launches += 8
        FakeEvent.clock[0] += 2.0  # each step takes 2 ms of fake device time

    K = 3
    steps_ms, kern_ms, launches = bench.timed_passes(_fake_torch(log), lib, step, K, "stream", flush, (0, 1))
    # the timed region: K steps, each after an L2 flush, none under profiling
    first_profile = next(i for i, e in enumerate(log) if e[0] == "profile_begin")
    timed = [e for e in log[:first_profile] if e[0] == "step"]
    assert len(timed) == K and all(not prof for _, prof in timed)
    flushes = [e for e in log[:first_profile] if e[0] == "flush"]
    assert len(flushes) == K
    assert steps_ms == [2.0] * K
    # only the timed steps' launches count
    assert launches == 8 * K
    # the kernel pass: the same K steps, profiled for the requested kinds, per-step averages returned
    assert log[first_profile] == ("profile_begin", (0, 1))
    passed = [e for e in log[first_profile:] if e[0] == "step"]
    assert len(passed) == K and all(prof for _, prof in passed)
    assert kern_ms == {"gemm_fwd": 6.0 / K, "gemm_bwd": 4.0 / K}


def test_timing_note_names_the_kernel_pass():
    note = bench.KERNEL_PASS_NOTE
    assert "second pass" in note and "whole steps" in note
