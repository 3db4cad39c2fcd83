"""CPU tests of the seeded input generator (no LoRA arithmetic involved)."""
import numpy as np
import pytest
import torch

from paper_2606_19528_gb300 import synth


def test_splitmix64_reference_values():
    # splitmix64 with state 0: the first outputs of the published generator
    # (state += 0x9E3779B97F4A7C15, then the finaliser) are
    # 0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F.
    k = 0
    got = [int(synth._mix(np.array([k + (i + 1) * int(synth.G) & (2**64 - 1)], dtype=np.uint64))[0])
           for i in range(3)]
    assert got == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    v = rng.standard_normal(100000) * 10.0 ** rng.integers(-20, 20, 100000)
    ours = synth.to_bf16_bits(v)
    theirs = torch.from_numpy(v.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, theirs)


def test_widening_is_exact():
    b = np.arange(0, 65536, dtype=np.uint16)
    b = b[(b & 0x7F80) != 0x7F80]  # finite values only
    f = synth.bf16_bits_to_f64(b)
    assert np.array_equal(synth.to_bf16_bits(f), b)


def test_distribution_moments():
    z = synth.bf16_bits_to_f64(synth.normal_bf16(synth.stream_key(0, 9, 9), (1 << 20,), 1.0))
    assert abs(z.mean()) < 5e-3 and abs(z.std() - 1.0) < 5e-3
    u = synth.bf16_bits_to_f64(synth.uniform_bf16(synth.stream_key(0, 9, 8), (1 << 20,), 0.5))
    assert u.min() >= -0.5 and u.max() <= 0.5 and abs(u.std() - 0.5 / np.sqrt(3)) < 2e-3


def test_streams_are_counter_based():
    key = synth.stream_key(0, 1, 2, 3)
    full = synth.uniform01(key, 1000)
    part = synth.uniform01(key, 100, offset=450)
    assert np.array_equal(full[450:550], part)
    assert synth.stream_key(0, 1, 2, 3) != synth.stream_key(0, 1, 2, 4)


@pytest.mark.skipif(synth._clib() is None, reason="C generator not built")
@pytest.mark.parametrize("n", [1, 2, 7, 100003])
def test_c_generator_matches_numpy(n):
    key = synth.stream_key(0, 4, 1, 2, 3)
    assert np.array_equal(synth.normal_bf16(key, (n,), 0.3, use_c=True),
                          synth.normal_bf16(key, (n,), 0.3, use_c=False))
    assert np.array_equal(synth.uniform_bf16(key, (n,), 0.05, use_c=True),
                          synth.uniform_bf16(key, (n,), 0.05, use_c=False))
