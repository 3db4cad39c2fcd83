"""Seeded synthetic inputs for the LoRA-linear workloads.

This module only draws random numbers and rounds them to bf16.  It holds none
of the LoRA arithmetic, so both the fp64 oracle (test side) and the CUDA path
consume the very same bytes without sharing any compute code.

Generator (counter based, so any slice can be drawn independently):

* mixing function: the splitmix64 finaliser of Steele, Lea and Flood
  ("Fast splittable pseudorandom number generators", OOPSLA 2014):
  z ^= z >> 30; z *= 0xBF58476D1CE4E5B9; z ^= z >> 27; z *= 0x94D049BB133111EB;
  z ^= z >> 31 (all mod 2**64).
* stream key: k0 = mix(seed + G), then k <- mix(k ^ (tag + G)) for each tag,
  G = 0x9E3779B97F4A7C15.
* element i of a stream: w = mix(k + (i + 1) * G);
  uniform u = ((w >> 11) + 0.5) * 2**-53, which lies in (0, 1).
* normals by the Box-Muller transform on consecutive pairs (u[2p], u[2p+1]):
  rho = sqrt(-2 ln u[2p]), z[2p] = rho cos(2 pi u[2p+1]), z[2p+1] = rho sin(...).
* every value is scaled in float64, rounded to float32 (round to nearest even)
  and then to bf16 (round to nearest even on the float32 bit pattern).

Distributions of the LoRA workloads: x, dy ~ N(0, 1); W ~ N(0, 1/d_in)
(variance 1/d_in); A ~ U(-1/sqrt(d_in), 1/sqrt(d_in)); B ~ N(0, 0.02**2)
(standard deviation 0.02), or B = 0 for the LoRA initialisation case.

4-bit base weights (the paper quantizes trained weights with a quantizer it
does not specify; here the codes and parameters are drawn directly): every
code byte is floor(256 u), so both 4-bit codes of a byte are uniform on
0..15 and independent; per (row, 64-column group) the scale is
s = s0 (0.5 + u1) with s0 = 2 sqrt(3) / (15 sqrt(d_in)) and the offset
b = -(7.5 + (2 u2 - 1)) s, so that s q + b has mean about 0 and variance
about 1/d_in, like W above; s and b are rounded to bf16.

LM-head inputs (the paper's XSum sequences and trained embeddings are not
available): hidden states h ~ N(0, 1) and embedding rows E ~ N(0, 1/d);
instruction-tuning masks, a prompt of non-trainable positions followed by a
trainable response; targets drawn cluster-first: the vocabulary is split
into clusters of consecutive ids, a target's cluster is Zipf-distributed
(rank r with weight r^-2.5, which puts |J| for 30 % of 2048 positions and
k = 500 near 9 k, inside the 2.7-14.4 k the paper reports for its top-k
runs) and its member uniform; the top-k table lists, for
token i, i itself, then the rest of its cluster in a seeded random order,
then tokens of the following clusters -- the locality that makes the union
of a sequence's top-k rows far smaller than the vocabulary.
"""
from __future__ import annotations

import ctypes
import math
import os

import numpy as np

G = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22

# tensor identifiers used as stream tags
TID_X, TID_W, TID_A, TID_B, TID_DY, TID_WQ, TID_WP = 1, 2, 3, 4, 5, 6, 7
TID_H, TID_E, TID_Y, TID_TOPK = 8, 9, 10, 11


def _mix(z: np.ndarray) -> np.ndarray:
    """splitmix64 finaliser, in place on a uint64 array (wraps mod 2**64)."""
    z ^= z >> np.uint64(30)
    z *= _M1
    z ^= z >> np.uint64(27)
    z *= _M2
    z ^= z >> np.uint64(31)
    return z


def stream_key(seed: int, *tags: int) -> int:
    """Key of the stream named by (seed, tags...)."""
    with np.errstate(over="ignore"):
        k = _mix(np.array([np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + G], dtype=np.uint64))
        for t in tags:
            k = _mix(k ^ (np.uint64(t & 0xFFFFFFFFFFFFFFFF) + G))
    return int(k[0])


def uniform01(key: int, n: int, offset: int = 0) -> np.ndarray:
    """Elements offset .. offset+n-1 of the stream `key` as float64 in (0, 1)."""
    out = np.empty(n, dtype=np.float64)
    k = np.uint64(key)
    with np.errstate(over="ignore"):
        for s in range(0, n, _CHUNK):
            e = min(n, s + _CHUNK)
            i = np.arange(offset + s + 1, offset + e + 1, dtype=np.uint64)
            w = _mix(k + i * G)
            out[s:e] = ((w >> np.uint64(11)).astype(np.float64) + 0.5) * (2.0 ** -53)
    return out


def normal(key: int, n: int) -> np.ndarray:
    """n standard normals from the stream `key` (Box-Muller on element pairs)."""
    m = (n + 1) // 2
    out = np.empty(2 * m, dtype=np.float64)
    for s in range(0, m, _CHUNK):
        e = min(m, s + _CHUNK)
        u = uniform01(key, 2 * (e - s), offset=2 * s)
        rho = np.sqrt(-2.0 * np.log(u[0::2]))
        ang = (2.0 * math.pi) * u[1::2]
        out[2 * s:2 * e:2] = rho * np.cos(ang)
        out[2 * s + 1:2 * e:2] = rho * np.sin(ang)
    return out[:n]


def to_bf16_bits(v: np.ndarray) -> np.ndarray:
    """float64 -> float32 (RNE) -> bf16 (RNE); returns the uint16 bit patterns."""
    f = np.ascontiguousarray(v, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    return u.astype(np.uint16).reshape(np.shape(v))


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    u = np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    u = np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32)


_CLIB = None
_CLIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "synth_c", "libsynth.so")


def _clib():
    """The multi-threaded C build of this generator (synth_c/synth.c), or None
    when it has not been built; both give the same bytes."""
    global _CLIB
    if _CLIB is None and os.path.exists(_CLIB_PATH):
        lib = ctypes.CDLL(_CLIB_PATH)
        for f in (lib.synth_normal_bf16, lib.synth_uniform_bf16):
            f.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p]
            f.restype = None
        _CLIB = lib
    return _CLIB


def normal_bf16(key: int, shape, std: float, use_c: bool = True) -> np.ndarray:
    """bf16 bits of std * N(0, 1) from the stream `key`."""
    n = int(np.prod(shape))
    lib = _clib() if use_c else None
    if lib is None:
        return to_bf16_bits(normal(key, n) * std).reshape(shape)
    out = np.empty(shape, dtype=np.uint16)
    lib.synth_normal_bf16(key, n, float(std), out.ctypes.data)
    return out


def uniform_bf16(key: int, shape, bound: float, use_c: bool = True) -> np.ndarray:
    """bf16 bits of U(-bound, bound) from the stream `key`."""
    n = int(np.prod(shape))
    lib = _clib() if use_c else None
    if lib is None:
        return to_bf16_bits((2.0 * uniform01(key, n) - 1.0) * bound).reshape(shape)
    out = np.empty(shape, dtype=np.uint16)
    lib.synth_uniform_bf16(key, n, float(bound), out.ctypes.data)
    return out


def gen_x(seed: int, cfg: int, group: int, layer: int, T: int, K: int) -> np.ndarray:
    """Activation x [T, K] ~ N(0, 1); `group` names the input buffer (projections
    that read the same decoder activation share one group)."""
    return normal_bf16(stream_key(seed, cfg, TID_X, group, layer), (T, K), 1.0)


def gen_dy(seed: int, cfg: int, proj: int, layer: int, T: int, N: int) -> np.ndarray:
    """Upstream gradient dy [T, N] ~ N(0, 1)."""
    return normal_bf16(stream_key(seed, cfg, TID_DY, proj, layer), (T, N), 1.0)


def gen_W(seed: int, cfg: int, proj: int, layer: int, N: int, K: int) -> np.ndarray:
    """Frozen base weight W [N, K] ~ N(0, 1/K) (nn.Linear layout, d_out x d_in)."""
    return normal_bf16(stream_key(seed, cfg, TID_W, proj, layer), (N, K), 1.0 / math.sqrt(K))


def gen_A(seed: int, cfg: int, proj: int, layer: int, r: int, K: int) -> np.ndarray:
    """LoRA down factor A [r, K] ~ U(-1/sqrt(K), 1/sqrt(K))."""
    return uniform_bf16(stream_key(seed, cfg, TID_A, proj, layer), (r, K), 1.0 / math.sqrt(K))


def gen_B(seed: int, cfg: int, proj: int, layer: int, N: int, r: int, zero: bool = False) -> np.ndarray:
    """LoRA up factor B [N, r] ~ N(0, 0.02**2), or all zeros (LoRA initialisation)."""
    if zero:
        return np.zeros((N, r), dtype=np.uint16)
    return normal_bf16(stream_key(seed, cfg, TID_B, proj, layer), (N, r), 0.02)


def gen_Wq(seed: int, cfg: int, proj: int, layer: int, N: int, K: int):
    """4-bit frozen weight of a [N, K] projection: (codes [N, K / 2] uint8,
    params [N, K / 64, 2] bf16 bits holding (s, b) per row and 64-column group)."""
    u = uniform01(stream_key(seed, cfg, TID_WQ, proj, layer), N * (K // 2))
    codes = np.minimum(np.floor(u * 256.0), 255.0).astype(np.uint8).reshape(N, K // 2)
    G_ = K // 64
    v = uniform01(stream_key(seed, cfg, TID_WP, proj, layer), 2 * N * G_).reshape(N, G_, 2)
    s0 = 2.0 * math.sqrt(3.0) / (15.0 * math.sqrt(K))
    sc = s0 * (0.5 + v[:, :, 0])
    sc_b = bf16_bits_to_f64(to_bf16_bits(sc))
    off = -(7.5 + (2.0 * v[:, :, 1] - 1.0)) * sc_b
    params = np.stack([to_bf16_bits(sc), to_bf16_bits(off)], axis=-1)
    return codes, params


def gen_h(seed: int, cfg: int, T: int, d: int) -> np.ndarray:
    """Hidden states h [T, d] ~ N(0, 1) entering the LM head."""
    return normal_bf16(stream_key(seed, cfg, TID_H), (T, d), 1.0)


def gen_E(seed: int, cfg: int, V: int, d: int) -> np.ndarray:
    """Frozen LM-head embedding E [V, d] ~ N(0, 1/d)."""
    return normal_bf16(stream_key(seed, cfg, TID_E), (V, d), 1.0 / math.sqrt(d))


def gen_mask(T: int, trainable_frac: float) -> np.ndarray:
    """Prompt then response: the last round(frac T) positions are trainable."""
    n = int(round(T * trainable_frac))
    m = np.zeros(T, dtype=np.uint8)
    if n > 0:
        m[T - n:] = 1
    return m


def gen_targets(seed: int, cfg: int, T: int, V: int, cluster: int, zipf: float = 2.5) -> np.ndarray:
    """Targets [T] int32: Zipf-distributed cluster, uniform member."""
    n_cl = (V + cluster - 1) // cluster
    u = uniform01(stream_key(seed, cfg, TID_Y), 2 * T).reshape(T, 2)
    w = np.arange(1, n_cl + 1, dtype=np.float64) ** -zipf
    cdf = np.cumsum(w) / w.sum()
    cl = np.minimum(np.searchsorted(cdf, u[:, 0]), n_cl - 1)
    size = np.minimum(cluster, V - cl * cluster)
    return (cl * cluster + np.minimum(np.floor(u[:, 1] * size), size - 1)).astype(np.int32)


def gen_topk_table(seed: int, cfg: int, V: int, k: int, cluster: int) -> np.ndarray:
    """Top-k table [V, k] int32 with cluster locality (see the module notes)."""
    out = np.empty((V, k), dtype=np.int32)
    key = stream_key(seed, cfg, TID_TOPK)
    n_cl = (V + cluster - 1) // cluster
    for c in range(n_cl):
        lo, hi = c * cluster, min(V, (c + 1) * cluster)
        members = np.arange(lo, hi)
        nxt = np.concatenate([np.arange(hi, V), np.arange(0, lo)])[: max(0, k - 1)]
        u = uniform01(key, (hi - lo) * (hi - lo), offset=lo * cluster).reshape(hi - lo, hi - lo)
        for r, i in enumerate(members):
            others = members[members != i]
            order = others[np.argsort(u[r, : len(others)], kind="stable")]
            row = np.concatenate([[i], order, nxt])[:k]
            out[i, : len(row)] = row
    return out
