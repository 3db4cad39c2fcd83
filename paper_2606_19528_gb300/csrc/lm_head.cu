// Reduced-vocabulary LM-head cross entropy with logits masking (Sections
// "Softmax Approximation" and "Logits Masking"): the index and element-wise
// passes around the two tensor-core contractions (fused_gemm.cu), which
// compute the logits of the trainable positions over the reduced vocabulary
// J and the hidden-state gradient.
//   vocab_mark      J = union of the trainable targets' first k top-k entries
//   vocab_count,    J and the trainable positions as ascending lists and
//   compact         their inverse maps (128 vocabulary segments counted, then
//                   compacted in parallel); the last block places each
//                   trainable target in J
//   gather_rows(2)  rows of h (trainable positions) and of E (J) made dense
//   ce_lse          per trainable position: log-sum-exp over J merged from the
//                   logits contraction's per-group partials, and its loss; the
//                   last block writes the per-position losses and their sum
//                   in a fixed order
//   ce_grad         G = softmax_J - onehot(target) in bf16 for the dh
//                   contraction, one streaming pass over the logits
//   ce_finish       the losses when no position is trainable
//   scatter_rows    dh rows of trainable positions, zeros elsewhere
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace lora {

namespace {

constexpr int kScanThreads = 1024;

// One block of 128 threads per position t: if t is trainable, flags[v] = 1
// for the k entries v of its target's table row (per 1024 entries, all loads
// of a thread issued before its stores).
constexpr int kMarkThreads = 128;

__global__ void __launch_bounds__(kMarkThreads) vocab_mark_kernel(const int32_t* __restrict__ targets,
                                                                  const uint8_t* __restrict__ mask, int T,
                                                                  const int32_t* __restrict__ topk, long long ld,
                                                                  int k, int V, uint8_t* __restrict__ flags,
                                                                  int32_t* __restrict__ counts) {
  griddep_wait();
  griddep_launch_dependents();
  for (int t = blockIdx.x; t < T; t += gridDim.x) {
    if (mask && !mask[t]) continue;
    const int y = targets[t];
    if (y < 0 || y >= V) {
      if (threadIdx.x == 0) counts[2] = 1;  // invalid target
      continue;
    }
    const int32_t* row = topk + (long long)y * ld;
    for (int j0 = 0; j0 < k; j0 += 8 * kMarkThreads) {
      int v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int j = j0 + threadIdx.x + q * kMarkThreads;
        v[q] = j < k ? row[j] : 0;
      }
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        if (j0 + threadIdx.x + q * kMarkThreads < k) {
          if (v[q] < 0 || v[q] >= V)
            counts[2] = 1;  // invalid table entry
          else
            flags[v[q]] = 1;
        }
      }
    }
  }
}

// Exclusive scan of one value per thread over the block; returns the total.
__device__ __forceinline__ int block_scan(int v, int* excl) {
  __shared__ int warp_tot[kScanThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_tot[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kScanThreads / 32 ? warp_tot[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < kScanThreads / 32) warp_tot[lane] = w;  // inclusive
  }
  __syncthreads();
  const int before = (warp > 0 ? warp_tot[warp - 1] : 0) + x - v;
  const int total = warp_tot[kScanThreads / 32 - 1];
  __syncthreads();
  *excl = before;
  return total;
}

// Ascending compaction of the set entries of [0, n) (flag(i) != 0) into
// list, with inv[i] = position in list or -1.  One block.
template <typename Flag>
__device__ int compact(int n, Flag flag, int32_t* list, int32_t* inv) {
  const int per = (n + kScanThreads - 1) / kScanThreads;
  const int b0 = min(n, (int)threadIdx.x * per), b1 = min(n, b0 + per);
  int cnt = 0;
  for (int i = b0; i < b1; ++i) cnt += flag(i) ? 1 : 0;
  int off;
  const int total = block_scan(cnt, &off);
  for (int i = b0; i < b1; ++i) {
    if (flag(i)) {
      list[off] = i;
      if (inv) inv[i] = off;
      ++off;
    } else if (inv) {
      inv[i] = -1;
    }
  }
  return total;
}

constexpr int kSegs = 128;  // vocabulary segments of the multi-block compaction

// Set flags per vocabulary segment (every token in full-vocabulary mode).
__global__ void __launch_bounds__(256) vocab_count_kernel(const uint8_t* __restrict__ flags, int V, int full,
                                                          int32_t* __restrict__ seg_counts) {
  griddep_wait();
  griddep_launch_dependents();
  const int seg = (V + kSegs - 1) / kSegs;
  const int b0 = min(V, (int)blockIdx.x * seg), b1 = min(V, b0 + seg);
  int c = 0;
  for (int i = b0 + threadIdx.x; i < b1; i += blockDim.x) c += (full || flags[i]) ? 1 : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
  __shared__ int wsum[8];
  if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int t = 0;
    for (int w = 0; w < 8; ++w) t += wsum[w];
    seg_counts[blockIdx.x] = t;
  }
}

// Blocks 0 .. kSegs-1: their segment of J (ascending) and pos; block kSegs:
// the trainable positions, their inverse map and the counts.
// The last block to finish also places each trainable target in J (ycol).
__device__ void ycol_rows(const int32_t* __restrict__ targets, const int32_t* tl, const int32_t* pos, int V,
                          int32_t* ycol, int32_t* counts) {
  const int nT = counts[0];
  for (int i = threadIdx.x; i < nT; i += blockDim.x) {
    const int y = targets[tl[i]];
    const int c = (y >= 0 && y < V) ? pos[y] : -1;
    if (c < 0) counts[2] = 1;  // a trainable target outside J (or out of range)
    ycol[i] = c < 0 ? 0 : c;
  }
}

__device__ void compact_part(const uint8_t* __restrict__ flags, int V, int full, const int32_t* __restrict__ seg_counts,
                             const uint8_t* __restrict__ mask, int T, int32_t* J, int32_t* pos, int32_t* tl,
                             int32_t* tpos, int32_t* counts, int* s_base_p) {
  int& s_base = *s_base_p;
  if (blockIdx.x < kSegs) {
    const int seg = (V + kSegs - 1) / kSegs;
    const int b0 = min(V, (int)blockIdx.x * seg), b1 = min(V, b0 + seg);
    if (threadIdx.x == 0) {
      int base = 0;
      for (int b = 0; b < (int)blockIdx.x; ++b) base += seg_counts[b];
      s_base = base;
    }
    __syncthreads();
    const int base = s_base;
    compact(b1 - b0, [&](int i) { return full || flags[b0 + i] != 0; }, J + base, nullptr);
    __syncthreads();
    // pos over the segment: J[base .. base + cnt) are ascending tokens of [b0, b1)
    for (int i = b0 + threadIdx.x; i < b1; i += kScanThreads) pos[i] = -1;
    __syncthreads();
    const int cnt = seg_counts[blockIdx.x];
    for (int q = threadIdx.x; q < cnt; q += kScanThreads) {
      J[base + q] += b0;  // compact wrote segment-relative indices
      pos[J[base + q]] = base + q;
    }
    return;
  }
  const int nT = compact(T, [&](int t) { return !mask || mask[t] != 0; }, tl, tpos);
  if (threadIdx.x == 0) {
    int nJ = 0;
    for (int b = 0; b < kSegs; ++b) nJ += seg_counts[b];
    counts[0] = nT;
    counts[1] = nJ;
  }
}

__global__ void __launch_bounds__(kScanThreads) compact_kernel(const uint8_t* __restrict__ flags, int V, int full,
                                                               const int32_t* __restrict__ seg_counts,
                                                               const uint8_t* __restrict__ mask, int T,
                                                               int32_t* J, int32_t* pos, int32_t* tl, int32_t* tpos,
                                                               int32_t* counts, const int32_t* __restrict__ targets,
                                                               int32_t* ycol, int32_t* done) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ int s_base, s_last;
  compact_part(flags, V, full, seg_counts, mask, T, J, pos, tl, tpos, counts, &s_base);
  // the last block to finish (every J, pos, tl written and visible) places the targets
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(done, 1) == (int)gridDim.x - 1;
  __syncthreads();
  if (s_last) {
    __threadfence();
    ycol_rows(targets, tl, pos, V, ycol, counts);
  }
}

__global__ void gather_rows_kernel(const __nv_bfloat16* __restrict__ src, long long ld,
                                   const int32_t* __restrict__ idx, int n, int d, __nv_bfloat16* __restrict__ dst) {
  griddep_wait();
  griddep_launch_dependents();
  const int vpr = d / 8;  // 16-byte vectors per row
  const long long total = (long long)n * vpr;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int i = (int)(e / vpr), v = (int)(e % vpr);
    const uint4* s = reinterpret_cast<const uint4*>(src + (long long)idx[i] * ld) + v;
    reinterpret_cast<uint4*>(dst + (long long)i * d)[v] = __ldg(s);
  }
}

// Two gathers in one launch (blockIdx.y selects the row set): one warp per
// row, four 16-byte loads in flight per lane.
__global__ void gather_rows2_kernel(const __nv_bfloat16* __restrict__ src_a, long long ld_a,
                                    const int32_t* __restrict__ idx_a, int n_a, __nv_bfloat16* __restrict__ dst_a,
                                    const __nv_bfloat16* __restrict__ src_b, long long ld_b,
                                    const int32_t* __restrict__ idx_b, int n_b, __nv_bfloat16* __restrict__ dst_b,
                                    int d) {
  griddep_wait();
  griddep_launch_dependents();
  const bool b = blockIdx.y == 1;
  const __nv_bfloat16* src = b ? src_b : src_a;
  const long long ld = b ? ld_b : ld_a;
  const int32_t* idx = b ? idx_b : idx_a;
  const int n = b ? n_b : n_a;
  __nv_bfloat16* dst = b ? dst_b : dst_a;
  const int vpr = d / 8, lane = threadIdx.x & 31;
  const int warps = gridDim.x * (blockDim.x >> 5);
  for (int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); i < n; i += warps) {
    const uint4* s = reinterpret_cast<const uint4*>(src + (long long)idx[i] * ld);
    uint4* o = reinterpret_cast<uint4*>(dst + (long long)i * d);
    for (int v0 = lane; v0 < vpr; v0 += 4 * 32) {
      uint4 q[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (v0 + u * 32 < vpr) q[u] = __ldg(s + v0 + u * 32);
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (v0 + u * 32 < vpr) o[v0 + u * 32] = q[u];
    }
  }
}

// Combine two (max, sum of exp(x - max)) pairs.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  if (m2 > m) {
    s = s * expf(m - m2) + s2;
    m = m2;
  } else if (m2 > -INFINITY) {
    s += s2 * expf(m2 - m);
  }
}

// Per-position losses (zeros off the trainable set) and their sum in a fixed
// order (fp64), by one block of 256 threads.
__device__ void finish_body(const float* rowloss, int nT, const int32_t* tpos, int T, float* token_loss,
                            float* loss) {
  __shared__ double part[256];
  if (token_loss)
    for (int t = threadIdx.x; t < T; t += blockDim.x) token_loss[t] = tpos[t] >= 0 ? rowloss[tpos[t]] : 0.f;
  double acc = 0.0;
  for (int i = threadIdx.x; i < nT; i += blockDim.x) acc += (double)rowloss[i];
  part[threadIdx.x] = acc;
  __syncthreads();
  for (int w = blockDim.x / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) *loss = (float)part[0];
}

// One block per trainable position i: its log-sum-exp over J from the logits
// contraction's per-group (max, sum of exp) partials, and its loss
// lse - z[i, ycol[i]].
__global__ void __launch_bounds__(256) ce_lse_kernel(const float2* __restrict__ part, int ld_part, int ngroups,
                                                     const float* __restrict__ Z, int ldz,
                                                     const int32_t* __restrict__ ycol, float* __restrict__ lse_out,
                                                     float* rowloss, const int32_t* __restrict__ tpos, int T,
                                                     float* __restrict__ token_loss, float* __restrict__ loss,
                                                     int* __restrict__ done) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ float sm[8], ss[8];
  const int i = blockIdx.x;
  const float2* pr = part + (long long)i * ld_part;
  float m = -INFINITY, s = 0.f;
  for (int g = threadIdx.x; g < ngroups; g += blockDim.x) {
    const float2 q = pr[g];
    lse_merge(m, s, q.x, q.y);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
    lse_merge(m, s, m2, s2);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    sm[warp] = m;
    ss[warp] = s;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float M = sm[0], S = ss[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) lse_merge(M, S, sm[w], ss[w]);
    const float lse = M + logf(S);
    lse_out[i] = lse;
    rowloss[i] = lse - Z[(long long)i * ldz + ycol[i]];
  }
  // the last block to finish (every rowloss written and visible) sums the losses
  __shared__ int s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(done, 1) == (int)gridDim.x - 1;
  __syncthreads();
  if (s_last) {
    __threadfence();
    finish_body(rowloss, (int)gridDim.x, tpos, T, token_loss, loss);
  }
}

// G[i, :] = bf16(exp(z - lse_i) - [j == ycol_i]) with zeros in [nJ, ldg): one
// read of the fp32 logits, 16-byte loads and 8-byte stores; work items are
// (row, 4096-column chunk) pairs over a grid-stride loop.
constexpr int kGradChunk = 4096;

__global__ void __launch_bounds__(256) ce_grad_kernel(const float* __restrict__ Z, int ldz, int nJ,
                                                      const int32_t* __restrict__ ycol,
                                                      const float* __restrict__ lse_in, int nT,
                                                      __nv_bfloat16* __restrict__ G, int ldg) {
  griddep_wait();
  griddep_launch_dependents();
  const int chunks = (ldg + kGradChunk - 1) / kGradChunk;
  const long long items = (long long)nT * chunks;
  for (long long e = blockIdx.x; e < items; e += gridDim.x) {
    const int i = (int)(e / chunks), c = (int)(e % chunks);
    const float lse = lse_in[i];
    const int yc = ycol[i];
    const float* z = Z + (long long)i * ldz;
    __nv_bfloat16* g = G + (long long)i * ldg;
    const int j_end = min(ldg, (c + 1) * kGradChunk);
#pragma unroll 4
    for (int j = c * kGradChunk + 4 * (int)threadIdx.x; j < j_end; j += 4 * (int)blockDim.x) {
      float4 q = make_float4(0.f, 0.f, 0.f, 0.f);
      if (j < nJ) q = __ldcs(reinterpret_cast<const float4*>(z + j));  // ldz >= j + 4: inside the row
      const float zv[4] = {q.x, q.y, q.z, q.w};
      float o[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) o[u] = j + u < nJ ? expf(zv[u] - lse) - (j + u == yc ? 1.f : 0.f) : 0.f;
      *reinterpret_cast<uint2*>(g + j) = make_uint2(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]));
    }
  }
}

__global__ void __launch_bounds__(256) ce_finish_kernel(const float* __restrict__ rowloss, int nT,
                                                        const int32_t* __restrict__ tpos, int T,
                                                        float* __restrict__ token_loss, float* __restrict__ loss) {
  griddep_wait();
  griddep_launch_dependents();
  finish_body(rowloss, nT, tpos, T, token_loss, loss);
}

__global__ void scatter_rows_kernel(const __nv_bfloat16* __restrict__ src, const int32_t* __restrict__ tpos, int T,
                                    int d, __nv_bfloat16* __restrict__ dst) {
  griddep_wait();
  griddep_launch_dependents();
  const int vpr = d / 8;
  const long long total = (long long)T * vpr;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int t = (int)(e / vpr), v = (int)(e % vpr);
    const int i = tpos[t];
    const uint4 x = i >= 0 ? reinterpret_cast<const uint4*>(src + (long long)i * d)[v] : make_uint4(0u, 0u, 0u, 0u);
    reinterpret_cast<uint4*>(dst + (long long)t * d)[v] = x;
  }
}

int grid_for(long long n, int threads, int cap) {
  long long b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > cap) b = cap;
  return (int)b;
}

}  // namespace

cudaError_t launch_ce_index(const CeIndex& a, cudaStream_t st) {
  cudaError_t e;
  if (a.topk) {
    e = launch_kernel(vocab_mark_kernel, dim3(std::min(a.T, 65535)), dim3(kMarkThreads), 0, st, 1, a.targets,
                      a.mask, a.T, a.topk, a.ld_topk, a.k, a.V, a.flags, a.counts);
    if (e != cudaSuccess) return e;
  }
  const int full = a.topk ? 0 : 1;
  e = launch_kernel(vocab_count_kernel, dim3(kSegs), dim3(256), 0, st, 1, (const uint8_t*)a.flags, a.V, full,
                    a.seg_counts);
  if (e != cudaSuccess) return e;
  return launch_kernel(compact_kernel, dim3(kSegs + 1), dim3(kScanThreads), 0, st, 1, (const uint8_t*)a.flags, a.V,
                       full, (const int32_t*)a.seg_counts, a.mask, a.T, a.J, a.pos, a.tl, a.tpos, a.counts, a.targets,
                       a.ycol, a.counts + 4);
}

cudaError_t launch_gather_rows2(const __nv_bfloat16* src_a, long long ld_a, const int32_t* idx_a, int n_a,
                                __nv_bfloat16* dst_a, const __nv_bfloat16* src_b, long long ld_b,
                                const int32_t* idx_b, int n_b, __nv_bfloat16* dst_b, int d, cudaStream_t st) {
  if (n_b <= 0) return launch_gather_rows(src_a, ld_a, idx_a, n_a, d, dst_a, st);
  if (n_a <= 0) return launch_gather_rows(src_b, ld_b, idx_b, n_b, d, dst_b, st);
  return launch_kernel(gather_rows2_kernel, dim3(grid_for(std::max(n_a, n_b), 8, 4096), 2), dim3(256), 0, st, 1,
                       src_a, ld_a, idx_a, n_a, dst_a, src_b, ld_b, idx_b, n_b, dst_b, d);
}

cudaError_t launch_gather_rows(const __nv_bfloat16* src, long long ld, const int32_t* idx, int n, int d,
                               __nv_bfloat16* dst, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  return launch_kernel(gather_rows_kernel, dim3(grid_for((long long)n * (d / 8), 256, 8192)), dim3(256), 0, st, 1,
                       src, ld, idx, n, d, dst);
}

cudaError_t launch_ce_rows(const float2* lse_part, int ld_part, const float* Z, int ldz, int nJ, const int32_t* ycol,
                           int nT, float* lse, float* rowloss, const int32_t* tpos, int T, float* token_loss,
                           float* loss, int* done, __nv_bfloat16* G, int ldg, int num_sms, cudaStream_t st) {
  if (nT <= 0) return cudaSuccess;
  const int ngroups = (nJ + gemm_lse_group() - 1) / gemm_lse_group();
  cudaError_t e = launch_kernel(ce_lse_kernel, dim3(nT), dim3(256), 0, st, 1, lse_part, ld_part, ngroups, Z, ldz,
                                ycol, lse, rowloss, tpos, T, token_loss, loss, done);
  if (e != cudaSuccess) return e;
  const long long items = (long long)nT * ((ldg + kGradChunk - 1) / kGradChunk);
  const int grid = (int)std::min<long long>(items, (long long)num_sms * 8);
  return launch_kernel(ce_grad_kernel, dim3(grid), dim3(256), 0, st, 1, Z, ldz, nJ, ycol, lse, nT, G, ldg);
}

cudaError_t launch_ce_finish(const float* rowloss, int nT, const int32_t* tpos, int T, float* token_loss,
                             float* loss, cudaStream_t st) {
  return launch_kernel(ce_finish_kernel, dim3(1), dim3(256), 0, st, 1, rowloss, nT, tpos, T, token_loss, loss);
}

cudaError_t launch_scatter_rows(const __nv_bfloat16* src, const int32_t* tpos, int T, int d, __nv_bfloat16* dst,
                                cudaStream_t st) {
  return launch_kernel(scatter_rows_kernel, dim3(grid_for((long long)T * (d / 8), 256, 8192)), dim3(256), 0, st, 1,
                       src, tpos, T, d, dst);
}

}  // namespace lora
