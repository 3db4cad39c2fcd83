"""CPU tests: the reduced-vocabulary cross-entropy oracle against its pins, and
planted mistakes (in copies of the oracle, on the CPU) that the pins must catch."""
import numpy as np
import pytest

from oracle import lm_head_oracle as O
from tests import lm_head_pins as P


@pytest.mark.parametrize("pin", P.PINS, ids=lambda p: p.__name__)
def test_ce_pin(pin):
    P.run_pin(pin, O.reduced_vocab, O.ce_forward_backward)


def _ce_full_vocab(h, E, targets, mask, J):
    return O.ce_forward_backward(h, E, targets, mask, np.arange(np.asarray(E).shape[0]))


def _ce_no_mask(h, E, targets, mask, J):
    return O.ce_forward_backward(h, E, targets, np.ones_like(np.asarray(mask, dtype=bool)), J)


def _ce_no_onehot(h, E, targets, mask, J):
    loss, per, dh = O.ce_forward_backward(h, E, targets, mask, J)
    E = np.asarray(E, dtype=np.float64)
    m = np.asarray(mask, dtype=bool)
    dh = dh.copy()
    dh[m] += E[np.asarray(targets)[m]]
    return loss, per, dh


def _ce_neg_grad(h, E, targets, mask, J):
    loss, per, dh = O.ce_forward_backward(h, E, targets, mask, J)
    return loss, per, -dh


def _vocab_k_minus_1(targets, mask, topk, k):
    return O.reduced_vocab(targets, mask, topk, max(1, k - 1))


def _vocab_all_targets(targets, mask, topk, k):
    return O.reduced_vocab(targets, np.ones_like(np.asarray(mask, dtype=bool)), topk, k)


MISTAKES = {
    "softmax_over_full_vocab": (O.reduced_vocab, _ce_full_vocab),
    "loss_over_all_positions": (O.reduced_vocab, _ce_no_mask),
    "dropped_onehot_term": (O.reduced_vocab, _ce_no_onehot),
    "gradient_sign": (O.reduced_vocab, _ce_neg_grad),
    "k_off_by_one": (_vocab_k_minus_1, O.ce_forward_backward),
    "vocab_from_untrainable_targets": (_vocab_all_targets, O.ce_forward_backward),
}


@pytest.mark.parametrize("name", sorted(MISTAKES))
def test_ce_pins_catch_planted_mistake(name):
    rv, ce = MISTAKES[name]
    failed = False
    for pin in P.PINS:
        try:
            P.run_pin(pin, rv, ce)
        except (AssertionError, KeyError):  # KeyError: a target outside the vocabulary it was given
            failed = True
    assert failed, f"no pin caught the planted mistake {name}"
