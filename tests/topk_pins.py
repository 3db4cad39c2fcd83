"""Pins that hold the top-k similarity-table oracle to facts other than its
own formulas.  Each pin takes a table function (E bits, k) -> [V, k] int32
(the oracle's, or a deliberately broken copy) and raises AssertionError when
it disagrees with:

* a hand-worked example, including ties (tests/golden), computed by hand;
* brute force on tiny inputs: the normalisation written out as scalar fp32
  steps in index order, similarities as Python sums, rows sorted with
  Python's sort on (-similarity, index);
* invariances: scaling a token's vector by a power of two leaves the table
  unchanged; relabelling the tokens relabels the table (no ties);
* the paper's remark that the first entry of row i is i itself (distinct
  directions).
"""
from __future__ import annotations

import json
import os

import numpy as np

from paper_2606_19528_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rand_E(rng, V, d):
    return synth.to_bf16_bits(rng.standard_normal((V, d)))


def pin_handworked(table):
    with open(os.path.join(GOLDEN, "topk_table_handworked_V4_d2.json")) as f:
        g = json.load(f)
    for E, want in ((g["E"], g["table_k4"]), (g["ties"]["E"], g["ties"]["table_k4"])):
        bits = synth.to_bf16_bits(np.array(E, dtype=np.float64))
        got = table(bits, 4)
        assert got.tolist() == want, (got.tolist(), want)
        assert table(bits, 2).tolist() == [row[:2] for row in want]


def _brute(bits, k):
    V, d = bits.shape
    vals = synth.bf16_bits_to_f64(bits)
    normed = []
    for i in range(V):
        s = np.float32(0.0)
        for c in range(d):
            x = np.float32(vals[i, c])
            s = np.float32(s + x * x)
        n = np.sqrt(s, dtype=np.float32)
        row = []
        for c in range(d):
            q = np.float32(0.0) if n == 0 else np.float32(np.float32(vals[i, c]) / n)
            row.append(float(synth.bf16_bits_to_f64(synth.to_bf16_bits(np.array([q], dtype=np.float64)))[0]))
        normed.append(row)
    out = []
    for i in range(V):
        sims = [(-sum(a * b for a, b in zip(normed[i], normed[j])), j) for j in range(V)]
        out.append([j for _, j in sorted(sims)[:k]])
    return out


def pin_brute_force(table, rng):
    for V, d, k in ((9, 5, 4), (12, 3, 12)):
        bits = _rand_E(rng, V, d)
        assert table(bits, k).tolist() == _brute(bits, k)


def pin_invariances(table, rng):
    V, d, k = 40, 16, 7
    bits = _rand_E(rng, V, d)
    base = table(bits, k)
    vals = synth.bf16_bits_to_f64(bits)
    scale = 2.0 ** rng.integers(-3, 4, size=(V, 1))
    assert np.array_equal(table(synth.to_bf16_bits(vals * scale), k), base)
    perm = rng.permutation(V)          # new token a is old token perm[a]
    inv = np.argsort(perm)
    relab = table(bits[perm], k)
    assert np.array_equal(relab, inv[base[perm]])


def pin_first_is_self(table, rng):
    bits = _rand_E(rng, 50, 8)
    t = table(bits, 5)
    assert np.array_equal(t[:, 0], np.arange(50))


PINS = (pin_handworked, pin_brute_force, pin_invariances, pin_first_is_self)


def run_pin(pin, table, seed=0):
    rng = np.random.default_rng(seed)
    if pin is pin_handworked:
        pin(table)
    else:
        pin(table, rng)
