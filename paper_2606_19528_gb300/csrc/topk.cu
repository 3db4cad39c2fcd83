// Top-k similarity table of a frozen embedding (Section "Softmax
// Approximation", "Choosing the Reduced Vocabulary Set"): token vectors are
// normalised, C = E~ E~^T holds the cosine similarities, and row i of the
// table lists the k most similar tokens in descending order (lower index
// first on ties).  The V x V matrix is never formed: rows are processed in
// chunks; a tcgen05 contraction (fused_gemm.cu, fp32 output) writes one
// chunk's similarities, and one CTA per row selects its top k from them.
//   normalize_rows  E~_i = bf16(E_i / ||E_i||), the sum of squares
//                   accumulated in fp32 in index order (squares of bf16 are
//                   exact), correctly rounded sqrt and division
//   topk_select     radix select on an order-preserving uint32 image of the
//                   similarities: 11-bit histograms (then 11, then 10 bits)
//                   until the candidates at or above the chosen prefix fit in
//                   shared memory, then a bitonic sort of the candidates on
//                   (similarity descending, index ascending)
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

// Order-preserving image of a float: larger value, larger key.
__device__ __forceinline__ uint32_t ord_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
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

__global__ void __launch_bounds__(kSelThreads) topk_select_kernel(const float* __restrict__ S, long long lds, int V,
                                                                  int k, int row0, int32_t* __restrict__ table,
                                                                  int* __restrict__ status) {
  griddep_wait();
  griddep_launch_dependents();
  extern __shared__ uint8_t smem_raw[];
  SelShared& sh = *reinterpret_cast<SelShared*>(smem_raw);
  const int r = blockIdx.x;
  const float* s = S + (long long)r * lds;  // lds is a multiple of 4: 16-byte aligned rows
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
    for (int j4 = threadIdx.x; j4 < V / 4; j4 += kSelThreads) {
      const float4 q = __ldg(reinterpret_cast<const float4*>(s) + j4);
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
  for (int j4 = threadIdx.x; j4 < V / 4; j4 += kSelThreads) {
    const float4 q = __ldcs(reinterpret_cast<const float4*>(s) + j4);  // last read of the row
    take(q.x, 4 * j4);
    take(q.y, 4 * j4 + 1);
    take(q.z, 4 * j4 + 2);
    take(q.w, 4 * j4 + 3);
  }
  for (int j = (V & ~3) + (int)threadIdx.x; j < V; j += kSelThreads) take(s[j], j);
  __syncthreads();
  const int n = sh.ncand;
  int p2 = 1;
  while (p2 < n) p2 <<= 1;
  for (int i = n + (int)threadIdx.x; i < p2; i += kSelThreads) {
    sh.ckey[i] = 0u;  // below every real key
    sh.cidx[i] = 0x7fffffff;
  }
  __syncthreads();
  // bitonic sort: "a before b" when a.key > b.key, or equal keys and a.idx < b.idx
  for (int size = 2; size <= p2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < p2 / 2; i += kSelThreads) {
        const int lo = 2 * i - (i & (stride - 1)), hi = lo + stride;
        const bool up = (lo & size) == 0;  // this run sorted "a before b"
        const uint32_t ka = sh.ckey[lo], kb = sh.ckey[hi];
        const int ia = sh.cidx[lo], ib = sh.cidx[hi];
        const bool b_first = kb > ka || (kb == ka && ib < ia);
        if (b_first == up) {
          sh.ckey[lo] = kb;
          sh.ckey[hi] = ka;
          sh.cidx[lo] = ib;
          sh.cidx[hi] = ia;
        }
      }
      __syncthreads();
    }
  }
  int32_t* out = table + (long long)(row0 + r) * k;
  for (int i = threadIdx.x; i < k; i += kSelThreads) out[i] = sh.cidx[i];
}

}  // namespace

cudaError_t launch_normalize_rows(const __nv_bfloat16* E, int V, int d, __nv_bfloat16* En, cudaStream_t st) {
  return launch_kernel(normalize_rows_kernel, dim3((V + 127) / 128), dim3(128), 0, st, 1, E, V, d, En);
}

cudaError_t launch_topk_select(const float* S, long long lds, int V, int k, int row0, int nrows, int32_t* table,
                               int* status, cudaStream_t st) {
  static bool attr_done = false;
  const int smem = (int)sizeof(SelShared);
  if (!attr_done) {
    cudaError_t e = cudaFuncSetAttribute(topk_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  return launch_kernel(topk_select_kernel, dim3(nrows), dim3(kSelThreads), smem, st, 1, S, lds, V, k, row0, table,
                       status);
}

int topk_max_k() { return kSelThreads; }

}  // namespace lora
