// Top-k similarity table of a frozen embedding (Section "Softmax
// Approximation", "Choosing the Reduced Vocabulary Set"): token vectors are
// normalised, C = E~ E~^T holds the cosine similarities, and row i of the
// table lists the k most similar tokens in descending order (lower index
// first on ties).  The V x V matrix is never formed.
//   normalize_rows      E~_i = bf16(E_i / ||E_i||), the sum of squares
//                       accumulated in fp32 in index order (squares of bf16
//                       are exact), correctly rounded sqrt and division
// Rows shorter than 32768 tokens (the host runs 512-row chunks):
//   topk_select         per row of a chunk's fp32 similarities (tcgen05
//                       contraction in fused_gemm.cu): radix select on an
//                       order-preserving uint32 image (11-bit histograms,
//                       then 11, then 10 bits) until the candidates at or
//                       above the chosen prefix fit in shared memory, then a
//                       sort on (similarity descending, index ascending); it
//                       also serves the longer rows' fallback
// Rows of at least 32768 tokens:
//   topk_gather_sample  8192 evenly spread tokens
//   topk_tau            each row's threshold from its similarities to them
//   (fused_gemm.cu)     the upper triangle of C, each value appended to the
//                       candidate lists of both its rows when it reaches
//                       their thresholds
//   topk_sort_warp,     each row's candidates sorted: a warp per list of up
//   topk_sort           to 1024 in registers, a block for longer lists
#include <algorithm>

#include "common.cuh"
#include "kernels.h"

namespace lora {

namespace {

constexpr int kSelThreads = 1024;
constexpr int kCap = 4096;  // candidates held in shared memory

__global__ void normalize_rows_kernel(const __nv_bfloat16* __restrict__ E, int V, int d,
                                      __nv_bfloat16* __restrict__ En) {
  griddep_wait();
  griddep_launch_dependents();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= V) return;
  const uint4* row = reinterpret_cast<const uint4*>(E + (long long)i * d);
  const int nv = d / 8;
  float s = 0.f;
  for (int v = 0; v < nv; ++v) {
    const uint4 q = __ldg(row + v);
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float lo = __uint_as_float(w[e] << 16), hi = __uint_as_float(w[e] & 0xFFFF0000u);
      s = __fadd_rn(s, __fmul_rn(lo, lo));  // each square is exact; index order
      s = __fadd_rn(s, __fmul_rn(hi, hi));
    }
  }
  const float n = __fsqrt_rn(s);
  uint4* out = reinterpret_cast<uint4*>(En + (long long)i * d);
  for (int v = 0; v < nv; ++v) {
    const uint4 q = __ldg(row + v);
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float lo = __uint_as_float(w[e] << 16), hi = __uint_as_float(w[e] & 0xFFFF0000u);
      const float a = n > 0.f ? __fdiv_rn(lo, n) : 0.f, b = n > 0.f ? __fdiv_rn(hi, n) : 0.f;
      o[e] = pack_bf16x2(a, b);
    }
    out[v] = make_uint4(o[0], o[1], o[2], o[3]);
  }
}


// Exclusive scan of one value per thread over the block; returns the total.
__device__ __forceinline__ int scan_block(int v, int* excl, int* warp_tot) {
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
    int w = warp_tot[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    warp_tot[lane] = w;
  }
  __syncthreads();
  *excl = (warp > 0 ? warp_tot[warp - 1] : 0) + x - v;
  const int total = warp_tot[31];
  __syncthreads();
  return total;
}

struct SelShared {
  int hist[2048];
  uint32_t ckey[kCap];
  int cidx[kCap];
  int warp_tot[32];
  int bin, above, ncand;
};

// Bin (of nbins, by descending bin index) where the k_rem-th largest falls,
// and the count in higher bins.
__device__ void find_bin(SelShared& sh, int nbins, int k_rem) {
  const int per = nbins / kSelThreads;  // 1 or 2
  const int t = threadIdx.x;
  int b0 = nbins - 1 - t * per;
  int local = 0;
  for (int q = 0; q < per; ++q) local += sh.hist[b0 - q];
  int excl;
  scan_block(local, &excl, sh.warp_tot);
  if (excl < k_rem && k_rem <= excl + local) {
    int acc = excl;
    for (int q = 0; q < per; ++q) {
      const int h = sh.hist[b0 - q];
      if (k_rem <= acc + h) {
        sh.bin = b0 - q;
        sh.above = acc;
        break;
      }
      acc += h;
    }
  }
  __syncthreads();
}

// A candidate as one 64-bit value, larger first: the order key above, the
// complement of the index below (equal keys: the lower index first).
__device__ __forceinline__ uint64_t pack_cand(uint32_t key, int idx) {
  return ((uint64_t)key << 32) | (uint32_t)(0xffffffffu - (uint32_t)idx);
}
__device__ __forceinline__ int cand_index(uint64_t v) { return (int)(0xffffffffu - (uint32_t)v); }

// Bitonic sort, descending, of p2 = kT * E packed candidates held in
// registers: slot e of thread t is position t + e * kT.  Strides below 32 are
// exchanged by warp shuffles, 32 .. kT / 2 through the shared buffer x (p2
// entries), kT and up within the thread (fully unrolled, so the slots stay in
// registers).  Every thread of the block takes part.
template <int kT, int E>
__device__ void bitonic_sort(uint64_t (&v)[E], uint64_t* x) {
  constexpr int p2 = kT * E;
  const int tid = kT == 32 ? (int)(threadIdx.x & 31) : (int)threadIdx.x;  // kT = 32: one warp, no barrier
  // fully unrolled: every stage's exchange form and masks are compile-time constants
#pragma unroll
  for (int size = 2; size <= p2; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      if (stride >= kT) {
#pragma unroll
        for (int lg = 0; (1 << lg) < E; ++lg) {
          if (stride == (kT << lg)) {
#pragma unroll
            for (int e = 0; e < E; ++e) {
              const int f = e | (1 << lg);
              if ((e & (1 << lg)) == 0 && f < E) {
                const bool up = ((tid + e * kT) & size) == 0;
                if ((v[f] > v[e]) == up) {
                  const uint64_t t = v[e];
                  v[e] = v[f];
                  v[f] = t;
                }
              }
            }
          }
        }
      } else {
        const bool via_smem = stride >= 32;
        if (via_smem) {
#pragma unroll
          for (int e = 0; e < E; ++e) x[tid + e * kT] = v[e];
          __syncthreads();
        }
#pragma unroll
        for (int e = 0; e < E; ++e) {
          const int p = tid + e * kT;
          const uint64_t q = via_smem ? x[p ^ stride] : __shfl_xor_sync(0xffffffffu, v[e], stride);
          const bool up = (p & size) == 0, lo = (p & stride) == 0;
          const bool q_first = q > v[e];
          // an ascending run keeps the first of the pair at the lower position
          if (lo ? q_first == up : q_first != up) v[e] = q;
        }
        if (via_smem) __syncthreads();
      }
    }
  }
}

// Loads n <= kT * E candidates (get(p) -> (key, index)), sorts them and writes
// the first k indices to out; padding sorts below every real candidate.
template <int kT, int E, typename Get>
__device__ void sort_write_e(Get get, int n, int k, uint64_t* x, int32_t* __restrict__ out) {
  const int tid = kT == 32 ? (int)(threadIdx.x & 31) : (int)threadIdx.x;
  uint64_t v[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int p = tid + e * kT;
    if (p < n) {
      const uint2 c = get(p);
      v[e] = pack_cand(c.x, (int)c.y);
    } else {
      v[e] = 0ull;
    }
  }
  if (kT > 32) __syncthreads();  // the candidates may live in the exchange buffer
  bitonic_sort<kT, E>(v, x);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const int p = tid + e * kT;
    if (p < k) out[p] = cand_index(v[e]);
  }
}

// Sorts the n candidates in shared memory (n <= kCap; the selection kernel's
// 1024 threads) and writes the first k indices to out.
__device__ void sort_and_write(SelShared& sh, int n, int k, int32_t* __restrict__ out) {
  auto get = [&](int p) { return make_uint2(sh.ckey[p], (uint32_t)sh.cidx[p]); };
  uint64_t* x = reinterpret_cast<uint64_t*>(sh.ckey);  // ckey and cidx together: 4096 x 8 bytes
  if (n <= kSelThreads)
    sort_write_e<kSelThreads, 1>(get, n, k, x, out);
  else if (n <= 2 * kSelThreads)
    sort_write_e<kSelThreads, 2>(get, n, k, x, out);
  else
    sort_write_e<kSelThreads, 4>(get, n, k, x, out);
}

// Sampled threshold for long rows: the r-th largest of kSample evenly spread
// row values (r sized so that about kOver * k of the row's values lie at or
// above it), found to 22 key bits by two histogram levels over the sample
// alone; then one streaming pass appends every value at or above that
// threshold, one ballot per 16-byte load and, for a warp with hits, one
// shared-memory atomic.  A value left out is strictly below every candidate,
// so when the candidates number between k and kCap they contain the exact
// top k.  Returns false (and the caller falls back to the full radix select)
// otherwise.
constexpr int kSample = 8 * kSelThreads;
constexpr int kSampleMinV = 4 * kSample;
constexpr float kOver = 1.6f;

// Rank of the sample value that sets the threshold: about kOver * k of a
// row's V values are expected at or above the rs-th largest of kSample.
__device__ __forceinline__ int sample_rank(int V, int k) {
  return min(kSample, max(1, (int)ceilf(kOver * (float)k * (float)kSample / (float)V)));
}

// The smallest value whose order key shares the top 22 bits of the rs-th
// largest of the block's kSample sample keys (8 per thread): two histogram
// levels of 11 bits over the sample.
__device__ float sample_threshold(SelShared& sh, const uint32_t* sk, int rs) {
  uint32_t prefix = 0;
  int r_rem = rs;
  for (int lvl = 0; lvl < 2; ++lvl) {
    for (int b = threadIdx.x; b < 2048; b += kSelThreads) sh.hist[b] = 0;
    __syncthreads();
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      if (lvl == 0)
        atomicAdd(&sh.hist[sk[e] >> 21], 1);
      else if ((sk[e] >> 21) == prefix)
        atomicAdd(&sh.hist[(sk[e] >> 10) & 2047u], 1);
    }
    __syncthreads();
    find_bin(sh, 2048, r_rem);
    prefix = (lvl == 0 ? 0u : prefix << 11) | (uint32_t)sh.bin;
    r_rem -= sh.above;
    __syncthreads();
  }
  const uint32_t key_lo = prefix << 10;
  return __uint_as_float((key_lo & 0x80000000u) ? (key_lo & 0x7fffffffu) : ~key_lo);
}

__device__ bool sampled_select(SelShared& sh, const float* __restrict__ s, int V, int k, int32_t* __restrict__ out) {
  const float4* s4 = reinterpret_cast<const float4*>(s);
  const int n4 = V / 4;
  const int lane = threadIdx.x & 31;
  uint32_t sk[8];  // this thread's sample keys, evenly spread over the row
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const float4 q = __ldg(s4 + (int)(((long long)(threadIdx.x + u * kSelThreads) * n4) / (2 * kSelThreads)));
    sk[4 * u + 0] = ord_key(q.x);
    sk[4 * u + 1] = ord_key(q.y);
    sk[4 * u + 2] = ord_key(q.z);
    sk[4 * u + 3] = ord_key(q.w);
  }
  const float tf = sample_threshold(sh, sk, sample_rank(V, k));
  if (threadIdx.x == 0) sh.ncand = 0;
  __syncthreads();
  // appends this lane's hits among its first nv values of q (positions j0 + e); whole warps call it
  auto append4 = [&](const float4 q, int nv, int j0) {
    const float f[4] = {q.x, q.y, q.z, q.w};
    const int c = (nv > 0 && f[0] >= tf) + (nv > 1 && f[1] >= tf) + (nv > 2 && f[2] >= tf) + (nv > 3 && f[3] >= tf);
    if (__ballot_sync(0xffffffffu, c > 0) == 0u) return;
    int x = c;  // inclusive scan of the hit counts over the warp
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    int base = 0;
    if (lane == 31) base = atomicAdd(&sh.ncand, x);
    int slot = __shfl_sync(0xffffffffu, base, 31) + x - c;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      if (e < nv && f[e] >= tf) {
        if (slot < kCap) {
          sh.ckey[slot] = ord_key(f[e]);
          sh.cidx[slot] = j0 + e;
        }
        ++slot;
      }
    }
  };
  // every thread runs the same iterations, so the ballots see whole warps
  for (int base4 = 0; base4 < n4; base4 += 4 * kSelThreads) {
    float4 q[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j4 = base4 + u * kSelThreads + (int)threadIdx.x;
      q[u] = j4 < n4 ? __ldcs(s4 + j4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j4 = base4 + u * kSelThreads + (int)threadIdx.x;
      append4(q[u], j4 < n4 ? 4 : 0, 4 * j4);
    }
  }
  if (threadIdx.x < 32) {  // the last V mod 4 values, one warp
    const int j = 4 * n4 + lane;
    append4(make_float4(j < V ? s[j] : 0.f, 0.f, 0.f, 0.f), j < V ? 1 : 0, j);
  }
  __syncthreads();
  const int n = sh.ncand;
  if (n < k || n > kCap) return false;  // uniform: read after the barrier
  sort_and_write(sh, n, k, out);
  return true;
}

__global__ void __launch_bounds__(kSelThreads, 2) topk_select_kernel(const float* __restrict__ S, long long lds, int V,
                                                                  int k, int row0, const int32_t* __restrict__ rows,
                                                                  int32_t* __restrict__ table,
                                                                  int* __restrict__ status) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ uint8_t smem_raw[];
  SelShared& sh = *reinterpret_cast<SelShared*>(smem_raw);
  const int r = blockIdx.x;
  const long long trow = rows ? rows[r] : row0 + r;  // table row of similarity row r
  const float* s = S + (long long)r * lds;  // lds is a multiple of 4: 16-byte aligned rows
  if (V >= kSampleMinV) {
    if (sampled_select(sh, s, V, k, table + trow * k)) return;
    __syncthreads();  // the fallback reuses the shared buffers
  }
  // levels: (shift of the level's digit, digit bits); the prefix so far selects candidates
  const int shifts[3] = {21, 10, 0}, bits[3] = {11, 11, 10};
  uint32_t prefix = 0;  // chosen digits so far, as key >> shift of the current level
  int k_rem = k, above_total = 0, lvl_found = -1;
  for (int lvl = 0; lvl < 3; ++lvl) {
    const int nb = 1 << bits[lvl], sh_ = shifts[lvl];
    for (int b = threadIdx.x; b < nb; b += kSelThreads) sh.hist[b] = 0;
    __syncthreads();
    const int hi_shift = sh_ + bits[lvl];  // bits above this level's digit
    auto count = [&](float f) {
      const uint32_t key = ord_key(f);
      if (lvl == 0 || (key >> hi_shift) == prefix) atomicAdd(&sh.hist[(key >> sh_) & (nb - 1)], 1);
    };
    const float4* s4 = reinterpret_cast<const float4*>(s);
    const int n4 = V / 4;
    int j4 = threadIdx.x;
    for (; j4 + 3 * kSelThreads < n4; j4 += 4 * kSelThreads) {  // four loads in flight per thread
      float4 q[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) q[u] = __ldg(s4 + j4 + u * kSelThreads);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        count(q[u].x);
        count(q[u].y);
        count(q[u].z);
        count(q[u].w);
      }
    }
    for (; j4 < n4; j4 += kSelThreads) {
      const float4 q = __ldg(s4 + j4);
      count(q.x);
      count(q.y);
      count(q.z);
      count(q.w);
    }
    for (int j = (V & ~3) + (int)threadIdx.x; j < V; j += kSelThreads) count(s[j]);
    __syncthreads();
    find_bin(sh, nb, k_rem);
    prefix = (lvl == 0 ? 0u : prefix << bits[lvl]) | (uint32_t)sh.bin;
    above_total += sh.above;
    k_rem -= sh.above;
    const int ncand = above_total + sh.hist[sh.bin];
    if (ncand <= kCap) {
      lvl_found = lvl;
      break;
    }
    __syncthreads();
  }
  if (lvl_found < 0) {
    if (threadIdx.x == 0) atomicCAS(status, 0, kStatusTopkTies);  // more ties at the k-th value than fit
    return;
  }
  // collect every key whose prefix at the chosen level is >= the chosen prefix
  const int sh_ = shifts[lvl_found];
  if (threadIdx.x == 0) sh.ncand = 0;
  __syncthreads();
  auto take = [&](float f, int j) {
    const uint32_t key = ord_key(f);
    if ((key >> sh_) >= prefix) {
      const int slot = atomicAdd(&sh.ncand, 1);
      sh.ckey[slot] = key;
      sh.cidx[slot] = j;
    }
  };
  {
    const float4* s4 = reinterpret_cast<const float4*>(s);
    const int n4 = V / 4;
    int j4 = threadIdx.x;
    for (; j4 + 3 * kSelThreads < n4; j4 += 4 * kSelThreads) {
      float4 q[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) q[u] = __ldcs(s4 + j4 + u * kSelThreads);  // last read of the row
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int j = 4 * (j4 + u * kSelThreads);
        take(q[u].x, j);
        take(q[u].y, j + 1);
        take(q[u].z, j + 2);
        take(q[u].w, j + 3);
      }
    }
    for (; j4 < n4; j4 += kSelThreads) {
      const float4 q = __ldcs(s4 + j4);
      take(q.x, 4 * j4);
      take(q.y, 4 * j4 + 1);
      take(q.z, 4 * j4 + 2);
      take(q.w, 4 * j4 + 3);
    }
  }
  for (int j = (V & ~3) + (int)threadIdx.x; j < V; j += kSelThreads) take(s[j], j);
  __syncthreads();
  sort_and_write(sh, sh.ncand, k, table + trow * k);
}

// Rows of the sample similarities Z [rows, kSample]: each row's threshold,
// the smallest sample value in the bin of a 2048-bin linear histogram over
// [min, max] of the row's sample that holds its rs-th largest value, so that
// between rs and rs + (that bin's count) sample values are at or above it.
// 256 threads, 32 values each.
constexpr int kTauThreads = 256;
constexpr int kTauPer = kSample / kTauThreads;

__global__ void __launch_bounds__(kTauThreads, 4) topk_tau_kernel(const float* __restrict__ Z, int V, int k,
                                                                float* __restrict__ tau) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ int hist[2048];
  __shared__ float red[2][kTauThreads / 32];
  __shared__ int s_bin;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float4* z4 = reinterpret_cast<const float4*>(Z + (long long)blockIdx.x * kSample);
  float v[kTauPer];
#pragma unroll
  for (int u = 0; u < kTauPer / 4; ++u) {
    const float4 q = __ldcs(z4 + tid + u * kTauThreads);
    v[4 * u] = q.x;
    v[4 * u + 1] = q.y;
    v[4 * u + 2] = q.z;
    v[4 * u + 3] = q.w;
  }
  float lo = v[0], hi = v[0];
#pragma unroll
  for (int e = 1; e < kTauPer; ++e) {
    lo = fminf(lo, v[e]);
    hi = fmaxf(hi, v[e]);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
  }
  for (int b = tid; b < 2048; b += kTauThreads) hist[b] = 0;
  if (lane == 0) {
    red[0][warp] = lo;
    red[1][warp] = hi;
  }
  __syncthreads();
  lo = red[0][0];
  hi = red[1][0];
#pragma unroll
  for (int w = 1; w < kTauThreads / 32; ++w) {
    lo = fminf(lo, red[0][w]);
    hi = fmaxf(hi, red[1][w]);
  }
  const float scale = hi > lo ? 2048.f / (hi - lo) : 0.f;
  auto bin_of = [&](float x) { return min(2047, max(0, (int)((x - lo) * scale))); };
#pragma unroll
  for (int e = 0; e < kTauPer; ++e) atomicAdd(&hist[bin_of(v[e])], 1);
  __syncthreads();
  // bins by descending index: thread t holds bins 2047 - 8t .. 2040 - 8t
  const int rs = sample_rank(V, k);
  int local = 0;
#pragma unroll
  for (int q = 0; q < 8; ++q) local += hist[2047 - 8 * tid - q];
  int x = local;  // inclusive scan over the block
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  __shared__ int wsum[kTauThreads / 32];
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  int excl = x - local;
  for (int w = 0; w < warp; ++w) excl += wsum[w];
  if (excl < rs && rs <= excl + local) {
    int acc = excl;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const int h = hist[2047 - 8 * tid - q];
      if (rs <= acc + h) {
        s_bin = 2047 - 8 * tid - q;
        break;
      }
      acc += h;
    }
  }
  __syncthreads();
  // the smallest sample value in the chosen bin
  const int bstar = s_bin;
  float m = INFINITY;
#pragma unroll
  for (int e = 0; e < kTauPer; ++e)
    if (bin_of(v[e]) == bstar) m = fminf(m, v[e]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fminf(m, __shfl_xor_sync(0xffffffffu, m, o));
  __syncthreads();
  if (lane == 0) red[0][warp] = m;
  __syncthreads();
  if (tid == 0) {
    float t = red[0][0];
    for (int w = 1; w < kTauThreads / 32; ++w) t = fminf(t, red[0][w]);
    tau[blockIdx.x] = t;
  }
}

// Each row's cnt[r] candidates (order key, token) appended by the similarity
// contraction; with k <= n <= cap they hold the exact top k.  One warp per row
// sorts lists of up to 1024 in registers (32 lanes x up to 32 slots: shuffles
// below stride 32, in-thread swaps above, no barrier); longer lists go to a
// list for the block sort below; rows outside [k, cap] join the fallback list.
constexpr int kWarpSortMax = 1024;
constexpr int kSortThreads = 256;

__global__ void __launch_bounds__(kSortThreads, 2) topk_sort_warp_kernel(
    const uint2* __restrict__ cand, const int* __restrict__ cnt, int cap, int k, int row0, int nrows,
    int32_t* __restrict__ table, int32_t* __restrict__ big_rows, int* __restrict__ big_count,
    int32_t* __restrict__ fail_rows, int* __restrict__ fail_count) {
  griddep_wait();
  griddep_launch_dependents();
  const int r = blockIdx.x * (kSortThreads / 32) + (int)(threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= nrows) return;  // whole warps
  const int n = cnt[r];
  if (n < k || n > cap || n > kCap) {
    if (lane == 0) fail_rows[atomicAdd(fail_count, 1)] = row0 + r;
    return;
  }
  if (n > kWarpSortMax) {
    if (lane == 0) big_rows[atomicAdd(big_count, 1)] = r;
    return;
  }
  const uint2* c = cand + (long long)r * cap;
  auto get = [&](int p) { return c[p]; };
  int32_t* out = table + (long long)(row0 + r) * k;
  if (n <= 128)
    sort_write_e<32, 4>(get, n, k, nullptr, out);
  else if (n <= 256)
    sort_write_e<32, 8>(get, n, k, nullptr, out);
  else if (n <= 512)
    sort_write_e<32, 16>(get, n, k, nullptr, out);
  else
    sort_write_e<32, 32>(get, n, k, nullptr, out);
}

// The rows the warp sort listed (more than 1024 candidates): one block of 256
// threads per row (up to 16 register slots each), rows taken from the list.
__global__ void __launch_bounds__(kSortThreads, 4) topk_sort_kernel(const uint2* __restrict__ cand,
                                                                   const int* __restrict__ cnt, int cap, int k,
                                                                   int row0, const int32_t* __restrict__ big_rows,
                                                                   const int* __restrict__ big_count,
                                                                   int32_t* __restrict__ table) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ uint64_t xs[kCap];
  const int nbig = *big_count;
  for (int i = blockIdx.x; i < nbig; i += gridDim.x) {
    const int r = big_rows[i];
    const int n = cnt[r];  // kWarpSortMax < n <= kCap
    const uint2* c = cand + (long long)r * cap;
    auto get = [&](int p) { return c[p]; };
    int32_t* out = table + (long long)(row0 + r) * k;
    if (n <= 8 * kSortThreads)
      sort_write_e<kSortThreads, 8>(get, n, k, xs, out);
    else
      sort_write_e<kSortThreads, 16>(get, n, k, xs, out);
    __syncthreads();  // the exchange buffer is free for the next row
  }
}

// Es[i, :] = En[floor(i * V / kSample), :]: the sample tokens, evenly spread.
__global__ void topk_gather_sample_kernel(const __nv_bfloat16* __restrict__ En, int V, int d,
                                          __nv_bfloat16* __restrict__ Es) {
  griddep_wait();
  griddep_launch_dependents();
  const int vpr = d / 8;
  const long long total = (long long)kSample * vpr;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int i = (int)(e / vpr), v = (int)(e % vpr);
    const long long src = (long long)i * V / kSample;
    reinterpret_cast<uint4*>(Es + (long long)i * d)[v] = reinterpret_cast<const uint4*>(En + src * d)[v];
  }
}

}  // namespace

cudaError_t launch_normalize_rows(const __nv_bfloat16* E, int V, int d, __nv_bfloat16* En, cudaStream_t st) {
  return launch_kernel(normalize_rows_kernel, dim3((V + 127) / 128), dim3(128), 0, st, 1, E, V, d, En);
}

// Sets the dynamic shared-memory size of the selection kernel (once per device).
cudaError_t sel_attrs() {
  static std::atomic<unsigned long long> attr_done{0};
  return set_smem_once(topk_select_kernel, (int)sizeof(SelShared), attr_done);
}

cudaError_t launch_topk_select(const float* S, long long lds, int V, int k, int row0, const int32_t* rows, int nrows,
                               int32_t* table, int* status, cudaStream_t st) {
  cudaError_t e = sel_attrs();
  if (e != cudaSuccess) return e;
  return launch_kernel(topk_select_kernel, dim3(nrows), dim3(kSelThreads), (int)sizeof(SelShared), st, 1, S, lds, V,
                       k, row0, rows, table, status);
}

cudaError_t launch_topk_tau(const float* Z, int V, int k, int nrows, float* tau, cudaStream_t st) {
  return launch_kernel(topk_tau_kernel, dim3(nrows), dim3(kTauThreads), 0, st, 1, Z, V, k, tau);
}

cudaError_t launch_topk_sort(const uint2* cand, int* cnt, int cap, int k, int row0, int nrows, int32_t* table,
                             int32_t* big_rows, int* big_count, int32_t* fail_rows, int* fail_count, int num_sms,
                             cudaStream_t st) {
  const int per = kSortThreads / 32;
  cudaError_t e = launch_kernel(topk_sort_warp_kernel, dim3((nrows + per - 1) / per), dim3(kSortThreads), 0, st, 1,
                                cand, (const int*)cnt, cap, k, row0, nrows, table, big_rows, big_count, fail_rows,
                                fail_count);
  if (e != cudaSuccess) return e;
  return launch_kernel(topk_sort_kernel, dim3(std::min(nrows, 4 * num_sms)), dim3(kSortThreads), 0, st, 1, cand,
                       (const int*)cnt, cap, k, row0, (const int32_t*)big_rows, (const int*)big_count, table);
}

cudaError_t launch_topk_gather_sample(const __nv_bfloat16* En, int V, int d, __nv_bfloat16* Es, int num_sms,
                                      cudaStream_t st) {
  return launch_kernel(topk_gather_sample_kernel, dim3(num_sms * 4), dim3(256), 0, st, 1, En, V, d, Es);
}

int topk_sample() { return kSample; }
int topk_sample_min_v() { return kSampleMinV; }
int topk_cap() { return kCap; }

int topk_max_k() { return kSelThreads; }

}  // namespace lora
