"""CPU tests: the top-k similarity-table oracle against its pins, and planted
mistakes (in copies of the oracle, on the CPU) that the pins must catch."""
import numpy as np
import pytest

from oracle import topk_oracle as O
from tests import topk_pins as P


@pytest.mark.parametrize("pin", P.PINS, ids=lambda p: p.__name__)
def test_topk_pin(pin):
    P.run_pin(pin, O.topk_table)


def _order(C, k, tie_high=False, ascending=False):
    V = C.shape[1]
    idx = -np.arange(V) if tie_high else np.arange(V)
    key = C if ascending else -C
    return np.stack([np.lexsort((idx, key[r]))[:k] for r in range(C.shape[0])]).astype(np.int32)


def _no_normalisation(bits, k):
    x = (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return _order(x @ x.T, k)


def _ascending(bits, k):
    En = O.normalize_rows(bits)
    return _order(O.similarities(En), k, ascending=True)


def _ties_high_first(bits, k):
    En = O.normalize_rows(bits)
    return _order(O.similarities(En), k, tie_high=True)


def _normalise_columns(bits, k):
    x = (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    n = np.linalg.norm(x, axis=0, keepdims=True)
    n[n == 0] = 1
    y = x / n
    return _order(y @ y.T, k)


def _k_off_by_one(bits, k):
    t = O.topk_table(bits, k)
    return np.concatenate([t[:, 1:], t[:, -1:]], axis=1)


MISTAKES = {"no_normalisation": _no_normalisation, "ascending": _ascending, "ties_high_first": _ties_high_first,
            "normalise_columns": _normalise_columns, "skips_first": _k_off_by_one}


@pytest.mark.parametrize("name", sorted(MISTAKES))
def test_topk_pins_catch_planted_mistake(name):
    failed = False
    for pin in P.PINS:
        try:
            P.run_pin(pin, MISTAKES[name])
        except AssertionError:
            failed = True
    assert failed, f"no pin caught the planted mistake {name}"
