"""fp64 CPU oracle of the reduced-vocabulary LM-head cross entropy with
logits masking.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports, links or
runs this module: only the tests, the smoke check and the benchmark's CPU
baseline arm use it.  It shares no code with the CUDA library.

What it computes (Section "Softmax Approximation" and Section "Logits
Masking").  Hidden states h [T, d] enter the frozen LM head E [V, d] (one
row per vocabulary token).  Targets y [T] and the trainable set T_set (a
boolean mask over token positions) come from the data.  The reduced
vocabulary is the union of the trainable targets' first k entries of the
top-k similarity table A [V, k_tab] (row i lists token indices in
descending similarity to i; its first entry is i itself):

    J = union over t in T_set of A[y_t, :k]        (all of [V] when k is None)

Logits are formed only for trainable positions (logits masking) and only
over J (softmax approximation):

    z_t[j] = h_t . E_j            t in T_set, j in J
    loss   = - sum_{t in T_set} log softmax_J(z_t)[y_t]

and, E being frozen, the only gradient is

    dh_t = sum_{j in J} (softmax_J(z_t)[j] - [j == y_t]) E_j   (t in T_set),   dh_t = 0 otherwise.

The paper writes the loss as the plain sum over trainable positions.  Every
function below is the plain definition in fp64 (numpy's matrix product and
the standard max-shifted log-sum-exp as the only library steps); pins that
hold it to other facts live in the test suite.
"""
from __future__ import annotations

import numpy as np


def reduced_vocab(targets, mask, topk, k):
    """Sorted J (int64): the union of the first k entries of the top-k table
    rows of the trainable targets (the full vocabulary is np.arange(V))."""
    targets = np.asarray(targets, dtype=np.int64)
    mask = np.asarray(mask, dtype=bool)
    rows = np.asarray(topk)[targets[mask], :k]
    return np.unique(rows.reshape(-1))


def ce_forward_backward(h, E, targets, mask, J):
    """Loss (fp64 scalar), per-position losses [T] (0 off T_set) and dh [T, d]."""
    h = np.asarray(h, dtype=np.float64)
    E = np.asarray(E, dtype=np.float64)
    targets = np.asarray(targets, dtype=np.int64)
    mask = np.asarray(mask, dtype=bool)
    J = np.asarray(J, dtype=np.int64)
    T = h.shape[0]
    rows = np.nonzero(mask)[0]
    pos = {int(j): i for i, j in enumerate(J)}
    ycol = np.array([pos[int(targets[t])] for t in rows], dtype=np.int64)
    EJ = E[J]
    z = h[rows] @ EJ.T                          # logits of trainable positions over J
    m = z.max(axis=1, keepdims=True)
    lse = (m + np.log(np.exp(z - m).sum(axis=1, keepdims=True)))[:, 0]
    per = np.zeros(T)
    per[rows] = lse - z[np.arange(len(rows)), ycol]
    p = np.exp(z - lse[:, None])
    p[np.arange(len(rows)), ycol] -= 1.0
    dh = np.zeros_like(h)
    dh[rows] = p @ EJ
    return float(per.sum()), per, dh
