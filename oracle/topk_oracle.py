"""CPU oracle of the top-k similarity table of a frozen embedding.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports, links or
runs this module: only the tests and the benchmark's CPU arms use it.  It
shares no code with the CUDA library.

What it computes (Section "Softmax Approximation", "Choosing the Reduced
Vocabulary Set").  The embedding's token vectors are normalised; the cosine
similarity of every pair of tokens is C = W~^T W~ (here with tokens as rows:
C = E~ E~^T); row i of the table lists the tokens by descending C[i, :]
and the first k entries are kept (int32).  The paper leaves ties
unspecified; the lower index goes first.

Precision.  The table is integer output decided by floating point, so the
normalisation follows the library's definition exactly: per token, the sum
of squares of its bf16 entries accumulated in fp32 in index order (each
square is exact in fp32), its fp32 square root, each entry divided by it in
fp32 and rounded to bf16 (round to nearest even); a zero row stays zero.
The similarities of those bf16 vectors are then exact here (fp64 sums of
products that are exact in fp64), and the order is decided on them; the
tensor-core sums on the GPU differ from them by at most d * 2^-24 (the
vectors have unit norm), which the parity tests account for.
"""
from __future__ import annotations

import numpy as np


def _bf16_rne(x32: np.ndarray) -> np.ndarray:
    u = np.ascontiguousarray(x32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return (u.astype(np.uint32) << np.uint32(16)).view(np.float32)


def normalize_rows(E_bits) -> np.ndarray:
    """bf16 bit patterns [V, d] -> the normalised rows as float32 values that are bf16."""
    x = (np.ascontiguousarray(E_bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)
    sq = x * x                                    # exact in fp32
    s = np.cumsum(sq, axis=1, dtype=np.float32)[:, -1]  # fp32, index order
    nrm = np.sqrt(s, dtype=np.float32)
    out = np.zeros_like(x)
    nz = nrm > 0
    out[nz] = _bf16_rne(x[nz] / nrm[nz, None])
    return out


def similarities(En: np.ndarray, rows=None) -> np.ndarray:
    """Exact cosine similarities of normalised rows (fp64 sums of exact products)."""
    A = En.astype(np.float64) if rows is None else En[rows].astype(np.float64)
    return A @ En.astype(np.float64).T


def topk_table(E_bits, k: int, rows=None) -> np.ndarray:
    """int32 [len(rows) or V, k]: each row's tokens by descending similarity, lower index first on ties."""
    En = normalize_rows(E_bits)
    C = similarities(En, rows)
    V = C.shape[1]
    idx = np.arange(V)
    out = np.empty((C.shape[0], k), dtype=np.int32)
    for r in range(C.shape[0]):
        order = np.lexsort((idx, -C[r]))
        out[r] = order[:k]
    return out
