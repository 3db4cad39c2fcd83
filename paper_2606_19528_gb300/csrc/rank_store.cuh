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

}  // namespace lora
