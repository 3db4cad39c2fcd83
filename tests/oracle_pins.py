"""Pins that hold the fp64 oracle to facts other than its own formulas.

Each pin takes the forward and backward functions under test (the oracle's,
or a deliberately broken copy in the mutation test) and raises
AssertionError when they disagree with:

* a hand-worked example on small integers (tests/golden), computed by hand;
* the chain rule applied entry by entry to the scalar forward sum
  (per-element derivatives, not the matrix formulas);
* central finite differences of L = <G, y>;  y is linear in each of x, A
  and B separately, so the central difference equals the derivative up to
  fp64 rounding;
* the merged-weight identity of LoRA: y = x (W + s B A)^T, dx = dy (W + s B A);
* the factorisation through the full weight gradient dW' = dy^T x:
  dB = s dW' A^T, dA = s B^T dW';
* the LoRA initialisation invariant: with B = 0 the adapter adds exact zeros,
  so y = x W^T and dx = dy W bit for bit, and dA = 0.
"""
from __future__ import annotations

import json
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = max(np.linalg.norm(b), 1e-300)
    return np.linalg.norm(a - b) / den


def rand_problem(rng, T, K, N, r, zero_B=False):
    x = rng.standard_normal((T, K))
    W = rng.standard_normal((N, K)) / np.sqrt(K)
    A = rng.uniform(-1, 1, (r, K)) / np.sqrt(K)
    B = np.zeros((N, r)) if zero_B else 0.5 * rng.standard_normal((N, r))
    dy = rng.standard_normal((T, N))
    return x, W, A, B, dy


def pin_handworked(fwd, bwd):
    with open(os.path.join(GOLDEN, "lora_handworked_T2_K3_N2_r1.json")) as f:
        g = json.load(f)
    a = {k: np.array(g[k], dtype=np.float64) for k in ("x", "W", "A", "B", "dy")}
    s = g["s"]
    y, u = fwd(a["x"], a["W"], a["A"], a["B"], s)
    dx, dA, dB, v = bwd(a["dy"], a["x"], a["W"], a["A"], a["B"], s)
    for name, got in (("u", u), ("y", y), ("v", v), ("dx", dx), ("dA", dA), ("dB", dB)):
        want = np.array(g[name], dtype=np.float64)
        assert got.shape == want.shape, (name, got.shape, want.shape)
        assert np.array_equal(got, want), (name, got, want)


def pin_chain_rule_entries(fwd, bwd, rng):
    """Tiny shapes; every gradient entry from per-element derivatives of
    y[t][n] = sum_k x[t][k] W[n][k] + s sum_j (sum_k x[t][k] A[j][k]) B[n][j]."""
    for (T, K, N, r) in ((1, 1, 1, 1), (3, 4, 2, 1), (5, 3, 4, 2), (8, 8, 8, 4), (2, 7, 5, 3)):
        s = float(rng.choice([0.5, 1.0, 2.0, 3.0]))
        x, W, A, B, dy = rand_problem(rng, T, K, N, r)
        y, _ = fwd(x, W, A, B, s)
        dx, dA, dB, _ = bwd(dy, x, W, A, B, s)
        yb = np.zeros((T, N))
        for t in range(T):
            for n in range(N):
                acc = 0.0
                for k in range(K):
                    acc += x[t][k] * W[n][k]
                for j in range(r):
                    uj = 0.0
                    for k in range(K):
                        uj += x[t][k] * A[j][k]
                    acc += s * uj * B[n][j]
                yb[t][n] = acc
        # d y[t][n] / d x[t][k] = W[n][k] + s sum_j B[n][j] A[j][k]
        dxb = np.zeros((T, K))
        for t in range(T):
            for k in range(K):
                acc = 0.0
                for n in range(N):
                    d = W[n][k]
                    for j in range(r):
                        d += s * B[n][j] * A[j][k]
                    acc += dy[t][n] * d
                dxb[t][k] = acc
        # d y[t][n] / d A[j][k] = s B[n][j] x[t][k]
        dAb = np.zeros((r, K))
        for j in range(r):
            for k in range(K):
                acc = 0.0
                for t in range(T):
                    for n in range(N):
                        acc += dy[t][n] * s * B[n][j] * x[t][k]
                dAb[j][k] = acc
        # d y[t][n] / d B[n][j] = s sum_k x[t][k] A[j][k]
        dBb = np.zeros((N, r))
        for n in range(N):
            for j in range(r):
                acc = 0.0
                for t in range(T):
                    uj = 0.0
                    for k in range(K):
                        uj += x[t][k] * A[j][k]
                    acc += dy[t][n] * s * uj
                dBb[n][j] = acc
        for name, got, want in (("y", y, yb), ("dx", dx, dxb), ("dA", dA, dAb), ("dB", dB, dBb)):
            assert _rel(got, want) <= 1e-12, (name, (T, K, N, r), _rel(got, want))


def pin_finite_differences(fwd, bwd, rng, n_samples=12):
    T, K, N, r, s = 6, 10, 7, 3, 2.0
    x, W, A, B, dy = rand_problem(rng, T, K, N, r)
    G = dy

    def L(x_, A_, B_):
        y, _ = fwd(x_, W, A_, B_, s)
        return float(np.sum(G * y))

    dx, dA, dB, _ = bwd(dy, x, W, A, B, s)
    h = 0.25
    for name, arr, grad in (("x", x, dx), ("A", A, dA), ("B", B, dB)):
        for _ in range(n_samples):
            idx = tuple(int(rng.integers(0, d)) for d in arr.shape)
            p, m = arr.copy(), arr.copy()
            p[idx] += h
            m[idx] -= h
            args_p = {"x": x, "A": A, "B": B}
            args_m = dict(args_p)
            args_p[name], args_m[name] = p, m
            fd = (L(args_p["x"], args_p["A"], args_p["B"]) - L(args_m["x"], args_m["A"], args_m["B"])) / (2 * h)
            assert abs(fd - grad[idx]) <= 1e-9 * max(1.0, abs(grad[idx])), (name, idx, fd, grad[idx])


def pin_merged_weight(fwd, bwd, rng):
    for (T, K, N, r, s) in ((16, 24, 40, 4, 2.0), (9, 33, 17, 8, 0.75), (32, 64, 48, 16, 2.0)):
        x, W, A, B, dy = rand_problem(rng, T, K, N, r)
        Wm = W + s * (B @ A)
        y, _ = fwd(x, W, A, B, s)
        dx, _, _, _ = bwd(dy, x, W, A, B, s)
        assert _rel(y, x @ Wm.T) <= 1e-12, ("y", _rel(y, x @ Wm.T))
        assert _rel(dx, dy @ Wm) <= 1e-12, ("dx", _rel(dx, dy @ Wm))


def pin_full_gradient_factorisation(fwd, bwd, rng):
    for (T, K, N, r, s) in ((16, 24, 40, 4, 2.0), (9, 33, 17, 8, 0.75), (32, 64, 48, 16, 2.0)):
        x, W, A, B, dy = rand_problem(rng, T, K, N, r)
        dWp = dy.T @ x
        _, dA, dB, _ = bwd(dy, x, W, A, B, s)
        assert _rel(dB, s * dWp @ A.T) <= 1e-12, ("dB", _rel(dB, s * dWp @ A.T))
        assert _rel(dA, s * B.T @ dWp) <= 1e-12, ("dA", _rel(dA, s * B.T @ dWp))


def pin_init_invariant(fwd, bwd, rng):
    for (T, K, N, r, s) in ((16, 24, 40, 4, 2.0), (32, 64, 48, 16, 2.0)):
        x, W, A, B, dy = rand_problem(rng, T, K, N, r, zero_B=True)
        y, _ = fwd(x, W, A, B, s)
        dx, dA, dB, _ = bwd(dy, x, W, A, B, s)
        assert np.array_equal(y, x @ W.T), "y != x W^T with B = 0"
        assert np.array_equal(dx, dy @ W), "dx != dy W with B = 0"
        assert not np.any(dA), "dA != 0 with B = 0"
        # dB is not zero at initialisation: it is s dy^T x A^T
        assert _rel(dB, s * dy.T @ (x @ A.T)) <= 1e-12


ALL_PINS = (pin_handworked, pin_chain_rule_entries, pin_finite_differences, pin_merged_weight,
            pin_full_gradient_factorisation, pin_init_invariant)


def run_pin(pin, fwd, bwd, seed=0):
    rng = np.random.default_rng(seed)
    if pin is pin_handworked:
        return pin(fwd, bwd)
    return pin(fwd, bwd, rng)


# ---------------------------------------------------------------- 4-bit dequantization (Algorithm 1)

def _q4_bytes_loop(codes_row_bytes, k):
    """Code of column k read bit by bit from the packed row (the interface's
    layout written out per element, independently of any vectorised unpack)."""
    m, rem = divmod(k, 8)
    i, hi = divmod(rem, 2)
    bit = 4 * i + 16 * hi
    byte = codes_row_bytes[4 * m + bit // 8]
    return (byte >> (bit % 8)) & 15


def pin_q4_handworked(unpack, dequant):
    with open(os.path.join(GOLDEN, "q4_dequant_handworked_N2_K128.json")) as f:
        g = json.load(f)
    codes = np.array(g["codes"], dtype=np.uint8)
    W = dequant(codes, np.array(g["s"]), np.array(g["b"]))
    assert np.array_equal(W, np.array(g["W"], dtype=np.float64)), W
    y = np.array(g["x"]) @ W.T
    assert np.array_equal(y, np.array(g["y"], dtype=np.float64)), y


def pin_q4_bitwise_layout(unpack, dequant, rng):
    """Every code of a random packed matrix equals the per-element bit read."""
    N, K = 3, 64
    codes = rng.integers(0, 256, size=(N, K // 2), dtype=np.uint8)
    q = unpack(codes)
    for n in range(N):
        row = [int(v) for v in codes[n]]
        for k in range(K):
            assert q[n, k] == _q4_bytes_loop(row, k), (n, k)


def pin_q4_affine_groups(unpack, dequant, rng):
    """s = 1, b = 0 gives the codes themselves; each group's (s, b) applies to
    exactly its 64 columns (checked one group at a time against scalar loops)."""
    N, K = 2, 192
    codes = rng.integers(0, 256, size=(N, K // 2), dtype=np.uint8)
    ones, zeros = np.ones((N, K // 64)), np.zeros((N, K // 64))
    W = dequant(codes, ones, zeros)
    for n in range(N):
        row = [int(v) for v in codes[n]]
        for k in range(K):
            assert W[n, k] == _q4_bytes_loop(row, k)
    s = rng.uniform(0.1, 2.0, (N, K // 64))
    b = rng.uniform(-1.0, 1.0, (N, K // 64))
    W = dequant(codes, s, b)
    for n in range(N):
        row = [int(v) for v in codes[n]]
        for k in range(K):
            g = k // 64
            assert abs(W[n, k] - (s[n, g] * _q4_bytes_loop(row, k) + b[n, g])) <= 1e-15 * (1 + abs(W[n, k]))


Q4_PINS = (pin_q4_handworked, pin_q4_bitwise_layout, pin_q4_affine_groups)


def run_q4_pin(pin, unpack, dequant, seed=0):
    rng = np.random.default_rng(seed)
    if pin is pin_q4_handworked:
        pin(unpack, dequant)
    else:
        pin(unpack, dequant, rng)
