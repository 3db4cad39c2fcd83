"""Pins that hold the fp64 LM-head cross-entropy oracle to facts other than
its own formulas.  Each pin takes the functions under test (the oracle's, or
a deliberately broken copy) and raises AssertionError when they disagree with:

* a hand-worked example (tests/golden), computed by hand, for the full and a
  reduced vocabulary;
* loss masking written out position by position: logits for every position,
  per-position loss and gradient, then zeroed off the trainable set -- the
  paper states that logits masking gives identical losses and gradients;
* central finite differences of the loss with respect to h;
* properties of the reduced vocabulary that the paper states: it contains
  every trainable target (the first entry of a table row is the token
  itself), it is the union of the rows' first k entries and no more.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def rand_case(rng, T=7, V=23, d=5, k=4, frac=0.6):
    h = rng.standard_normal((T, d))
    E = rng.standard_normal((V, d))
    targets = rng.integers(0, V, T)
    mask = rng.random(T) < frac
    mask[0] = True
    topk = np.empty((V, V), dtype=np.int64)
    for i in range(V):
        rest = [j for j in rng.permutation(V) if j != i]
        topk[i] = [i] + rest
    return h, E, targets, mask, topk, k


def pin_handworked(reduced_vocab, ce):
    with open(os.path.join(GOLDEN, "ce_reduced_vocab_handworked_V4_d2_T3.json")) as f:
        g = json.load(f)
    h, E = np.array(g["h"], dtype=np.float64), np.array(g["E"], dtype=np.float64)
    targets, mask, topk = np.array(g["targets"]), np.array(g["mask"], dtype=bool), np.array(g["topk"])
    for case in g["cases"]:
        J = reduced_vocab(targets, mask, topk, case["k"])
        assert list(J) == case["J"], (J, case["J"])
        loss, per, dh = ce(h, E, targets, mask, J)
        assert abs(loss - math.log(case["loss_ln"])) < 1e-12, (loss, case["loss_ln"])
        assert np.allclose(per, [math.log(v) for v in case["per_ln"]], rtol=0, atol=1e-12), per
        assert np.allclose(dh, np.array(case["dh"]), rtol=0, atol=1e-12), dh


def _loss_masking_loops(h, E, targets, mask, J):
    """Every position's logits over J and its loss and gradient, one scalar at
    a time, then the mask applied to the loss and to the gradient."""
    T, d = h.shape
    total = 0.0
    per = [0.0] * T
    dh = np.zeros((T, d))
    for t in range(T):
        z = [sum(h[t, c] * E[j, c] for c in range(d)) for j in J]
        m = max(z)
        s = sum(math.exp(v - m) for v in z)
        lse = m + math.log(s)
        zy = sum(h[t, c] * E[targets[t], c] for c in range(d))
        lt = lse - zy
        g = np.zeros(d)
        for jj, j in enumerate(J):
            pj = math.exp(z[jj] - lse) - (1.0 if j == targets[t] else 0.0)
            g += pj * E[j]
        keep = 1.0 if mask[t] else 0.0
        per[t] = keep * lt
        total += keep * lt
        dh[t] = keep * g
    return total, np.array(per), dh


def pin_loss_masking_equivalence(reduced_vocab, ce, rng):
    h, E, targets, mask, topk, k = rand_case(rng)
    J = reduced_vocab(targets, mask, topk, k)
    loss, per, dh = ce(h, E, targets, mask, J)
    l2, p2, d2 = _loss_masking_loops(h, E, targets, mask, J)
    assert abs(loss - l2) <= 1e-10 * max(1.0, abs(l2)), (loss, l2)
    assert np.allclose(per, p2, rtol=1e-10, atol=1e-12)
    assert np.allclose(dh, d2, rtol=1e-10, atol=1e-12)


def pin_finite_differences(reduced_vocab, ce, rng, eps=1e-5):
    h, E, targets, mask, topk, k = rand_case(rng)
    J = reduced_vocab(targets, mask, topk, k)
    _, _, dh = ce(h, E, targets, mask, J)
    for _ in range(10):
        t, c = int(rng.integers(0, h.shape[0])), int(rng.integers(0, h.shape[1]))
        hp, hm = h.copy(), h.copy()
        hp[t, c] += eps
        hm[t, c] -= eps
        num = (ce(hp, E, targets, mask, J)[0] - ce(hm, E, targets, mask, J)[0]) / (2 * eps)
        assert abs(num - dh[t, c]) <= 1e-6 * max(1.0, abs(num)), (t, c, num, dh[t, c])


def pin_vocab_properties(reduced_vocab, ce, rng):
    h, E, targets, mask, topk, k = rand_case(rng, V=40, k=3)
    J = set(int(j) for j in reduced_vocab(targets, mask, topk, k))
    want = set()
    for t in range(len(targets)):
        if mask[t]:
            want.update(int(v) for v in topk[targets[t], :k])
            assert int(targets[t]) in J
    assert J == want, (sorted(J), sorted(want))


PINS = (pin_handworked, pin_loss_masking_equivalence, pin_finite_differences, pin_vocab_properties)


def run_pin(pin, reduced_vocab, ce, seed=0):
    rng = np.random.default_rng(seed)
    if pin is pin_handworked:
        pin(reduced_vocab, ce)
    else:
        pin(reduced_vocab, ce, rng)
