// Output side of the rank-r products, shared by their tensor-core kernels and
// the partial-sum pass.  A problem's rank side is the concatenation of up to
// kMaxRankBlocks projections' blocks, each padded to 8 columns.
#pragma once

#include "common.cuh"
#include "kernels.h"

namespace lora {

__device__ __forceinline__ int pad8(int r) { return (r + 7) & ~7; }

// Block of concatenated rank column j and the column within it (-1 past the last block).
__device__ __forceinline__ int find_block(const int* rw, int nblk, int j, int* jj) {
  int off = 0;
#pragma unroll
  for (int b = 0; b < kMaxRankBlocks; ++b) {
    if (b < nblk) {
      const int w = pad8(rw[b]);
      if (j < off + w) {
        *jj = j - off;
        return b;
      }
      off += w;
    }
  }
  return -1;
}

// Row product element (t, j), unscaled: bf16 of scale * v into out [T, ld_out],
// the optional copy out2 and the optional transposed copy outT [pad8(r), T];
// the padding columns j in [r, pad8(r)) are written as zeros.
__device__ __forceinline__ void row_store(const RowProb& P, int t, int j, float v) {
  int jj;
  const int b = find_block(P.rw, P.nblk, j, &jj);
  if (b < 0) return;
  const __nv_bfloat16 o = __float2bfloat16_rn(jj < P.rw[b] ? P.scale * v : 0.f);
  if (jj < P.ld_out[b]) P.out[b][(size_t)t * P.ld_out[b] + jj] = o;
  if (P.out2[b] != nullptr && jj < P.ld_out2[b]) P.out2[b][(size_t)t * P.ld_out2[b] + jj] = o;
  if (P.outT[b] != nullptr) P.outT[b][(size_t)jj * P.T + t] = o;
}

// Column product element (c, j) in fp32: out [C, r] (out_cr) or [r, C].
__device__ __forceinline__ void col_store(const ColProb& P, int c, int j, float v) {
  int jj;
  const int b = find_block(P.rs, P.nblk, j, &jj);
  if (b < 0 || jj >= P.rs[b]) return;
  if (P.out_cr)
    P.out[b][(size_t)c * P.rs[b] + jj] = v;
  else
    P.out[b][(size_t)jj * P.C + c] = v;
}

__device__ __forceinline__ bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Row product elements (t, j .. j + 7), j a multiple of 8 (so one rank block
// holds all eight): as row_store, with one 16-byte store per output row where
// its layout allows.
__device__ __forceinline__ void row_store8(const RowProb& P, int t, int j, const uint32_t* v) {
  int jj;
  const int b = find_block(P.rw, P.nblk, j, &jj);
  if (b < 0) return;
  uint32_t w[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float a = jj + 2 * e < P.rw[b] ? P.scale * __uint_as_float(v[2 * e]) : 0.f;
    const float c = jj + 2 * e + 1 < P.rw[b] ? P.scale * __uint_as_float(v[2 * e + 1]) : 0.f;
    w[e] = pack_bf16x2(a, c);
  }
  const __nv_bfloat16* o = reinterpret_cast<const __nv_bfloat16*>(w);
  __nv_bfloat16* dsts[2] = {P.out[b], P.out2[b]};
  const int lds[2] = {P.ld_out[b], P.ld_out2[b]};
#pragma unroll
  for (int k = 0; k < 2; ++k) {
    if (dsts[k] == nullptr) continue;
    __nv_bfloat16* d = dsts[k] + (size_t)t * lds[k] + jj;
    if ((lds[k] & 7) == 0 && jj + 8 <= lds[k] && aligned16(dsts[k])) {
      *reinterpret_cast<uint4*>(d) = make_uint4(w[0], w[1], w[2], w[3]);
    } else {
      for (int e = 0; e < 8 && jj + e < lds[k]; ++e) d[e] = o[e];
    }
  }
  if (P.outT[b] != nullptr)
#pragma unroll
    for (int e = 0; e < 8; ++e) P.outT[b][(size_t)(jj + e) * P.T + t] = o[e];
}

// Column product elements (c, j .. j + 7), j a multiple of 8: as col_store,
// with 16-byte stores into the [C, r] layout where it allows.
__device__ __forceinline__ void col_store8(const ColProb& P, int c, int j, const uint32_t* v) {
  int jj;
  const int b = find_block(P.rs, P.nblk, j, &jj);
  if (b < 0) return;
  const int n = min(8, P.rs[b] - jj);
  if (n <= 0) return;
  if (P.out_cr) {
    float* d = P.out[b] + (size_t)c * P.rs[b] + jj;
    if (n == 8 && (P.rs[b] & 3) == 0 && aligned16(P.out[b])) {
      reinterpret_cast<float4*>(d)[0] =
          make_float4(__uint_as_float(v[0]), __uint_as_float(v[1]), __uint_as_float(v[2]), __uint_as_float(v[3]));
      reinterpret_cast<float4*>(d)[1] =
          make_float4(__uint_as_float(v[4]), __uint_as_float(v[5]), __uint_as_float(v[6]), __uint_as_float(v[7]));
    } else {
      for (int e = 0; e < n; ++e) d[e] = __uint_as_float(v[e]);
    }
  } else {
    for (int e = 0; e < n; ++e) P.out[b][(size_t)(jj + e) * P.C + c] = __uint_as_float(v[e]);
  }
}

}  // namespace lora
