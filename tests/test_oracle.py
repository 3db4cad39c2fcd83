"""CPU tests: the fp64 oracle against its pins, and planted mistakes that the
pins must catch (mistakes are planted in copies of the oracle, on the CPU)."""
import numpy as np
import pytest

import oracle
from oracle import lora_oracle as O
from tests import oracle_pins as P


@pytest.mark.parametrize("pin", P.ALL_PINS, ids=lambda p: p.__name__)
def test_oracle_pin(pin):
    P.run_pin(pin, oracle.lora_forward, oracle.lora_backward)


def test_rows_helpers_match_full():
    rng = np.random.default_rng(3)
    x, W, A, B, dy = P.rand_problem(rng, 20, 12, 9, 3)
    s = 2.0
    y, _ = oracle.lora_forward(x, W, A, B, s)
    dx, dA, dB, _ = oracle.lora_backward(dy, x, W, A, B, s)
    rows = np.array([0, 5, 19, 7])
    assert np.allclose(oracle.lora_forward_rows(rows, x, W, A, B, s), y[rows], rtol=1e-13, atol=1e-13)
    assert np.allclose(oracle.lora_backward_dx_rows(rows, dy, W, A, B, s), dx[rows], rtol=1e-13, atol=1e-13)
    dA2, dB2 = oracle.lora_adapter_grads(dy, x, A, B, s)
    assert np.allclose(dA2, dA, rtol=1e-13, atol=1e-12) and np.allclose(dB2, dB, rtol=1e-13, atol=1e-12)


# ---- planted mistakes: each must make at least one pin fail -----------------

def _fwd_drop_scale(x, W, A, B, s):
    return oracle.lora_forward(x, W, A, B, 1.0)


def _fwd_wrong_sign(x, W, A, B, s):
    y, u = oracle.lora_forward(x, W, A, B, s)
    return y - 2 * s * (u @ np.asarray(B, float).T), u


def _fwd_transposed_B(x, W, A, B, s):
    x, W, A, B = (np.asarray(a, float) for a in (x, W, A, B))
    u = x @ A.T
    Bt = B.reshape(B.shape[1], B.shape[0])  # reinterpreted storage: a layout slip
    return x @ W.T + s * (u @ Bt), u


def _bwd_drop_adapter_dx(dy, x, W, A, B, s):
    dx, dA, dB, v = oracle.lora_backward(dy, x, W, A, B, s)
    return np.asarray(dy, float) @ np.asarray(W, float), dA, dB, v


def _bwd_dB_no_scale(dy, x, W, A, B, s):
    dx, dA, dB, v = oracle.lora_backward(dy, x, W, A, B, s)
    return dx, dA, dB / s, v


def _bwd_dA_uses_u(dy, x, W, A, B, s):
    dx, dA, dB, v = oracle.lora_backward(dy, x, W, A, B, s)
    u = np.asarray(x, float) @ np.asarray(A, float).T
    return dx, s * (u.T @ np.asarray(x, float)), dB, v


def _bwd_dx_wrong_index(dy, x, W, A, B, s):
    dx, dA, dB, v = oracle.lora_backward(dy, x, W, A, B, s)
    return dx[::-1].copy(), dA, dB, v


def _bwd_sign_dA(dy, x, W, A, B, s):
    dx, dA, dB, v = oracle.lora_backward(dy, x, W, A, B, s)
    return dx, -dA, dB, v


MUTANTS = [
    ("fwd_drop_scale", _fwd_drop_scale, oracle.lora_backward),
    ("fwd_wrong_sign", _fwd_wrong_sign, oracle.lora_backward),
    ("fwd_transposed_B", _fwd_transposed_B, oracle.lora_backward),
    ("bwd_drop_adapter_dx", oracle.lora_forward, _bwd_drop_adapter_dx),
    ("bwd_dB_no_scale", oracle.lora_forward, _bwd_dB_no_scale),
    ("bwd_dA_uses_u", oracle.lora_forward, _bwd_dA_uses_u),
    ("bwd_dx_wrong_index", oracle.lora_forward, _bwd_dx_wrong_index),
    ("bwd_sign_dA", oracle.lora_forward, _bwd_sign_dA),
]


@pytest.mark.parametrize("name,fwd,bwd", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(name, fwd, bwd):
    failed = []
    for pin in P.ALL_PINS:
        try:
            P.run_pin(pin, fwd, bwd)
        except (AssertionError, ValueError):
            failed.append(pin.__name__)
    assert failed, f"no pin caught the planted mistake {name}"


# ---- 4-bit dequantization -----------------------------------------------------

@pytest.mark.parametrize("pin", P.Q4_PINS, ids=lambda p: p.__name__)
def test_q4_pin(pin):
    P.run_q4_pin(pin, O.unpack_q4, O.dequant_q4)


def _unpack_swapped_halves(codes):
    q = O.unpack_q4(codes)
    out = q.copy()
    out[:, 0::2], out[:, 1::2] = q[:, 1::2], q[:, 0::2]
    return out


def _unpack_nibble_order(codes):
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    lo, hi = c & 15, c >> 4
    return np.stack([lo, hi], axis=-1).reshape(c.shape[0], -1).astype(np.int64)


def _dequant_from(unpack):
    def dq(codes, s, b):
        q = unpack(codes).astype(np.float64)
        g = np.arange(q.shape[1]) // 64
        return np.asarray(s, dtype=np.float64)[:, g] * q + np.asarray(b, dtype=np.float64)[:, g]
    return dq


def _dequant_group_32(codes, s, b):
    q = O.unpack_q4(codes).astype(np.float64)
    g = np.minimum(np.arange(q.shape[1]) // 32, np.asarray(s).shape[1] - 1)
    return np.asarray(s, dtype=np.float64)[:, g] * q + np.asarray(b, dtype=np.float64)[:, g]


def _dequant_no_offset(codes, s, b):
    return O.dequant_q4(codes, s, np.zeros_like(np.asarray(b, dtype=np.float64)))


Q4_MISTAKES = {
    "swapped_pair_halves": (_unpack_swapped_halves, _dequant_from(_unpack_swapped_halves)),
    "plain_nibble_order": (_unpack_nibble_order, _dequant_from(_unpack_nibble_order)),
    "group_of_32": (O.unpack_q4, _dequant_group_32),
    "dropped_offset": (O.unpack_q4, _dequant_no_offset),
}


@pytest.mark.parametrize("name", sorted(Q4_MISTAKES))
def test_q4_pins_catch_planted_mistake(name):
    unpack, dequant = Q4_MISTAKES[name]
    failed = False
    for pin in P.Q4_PINS:
        try:
            P.run_q4_pin(pin, unpack, dequant)
        except AssertionError:
            failed = True
    assert failed, f"no pin caught the planted mistake {name}"
