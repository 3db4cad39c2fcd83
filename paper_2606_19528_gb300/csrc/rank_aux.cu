// Small passes around the rank-r products (those run on the tensor cores,
// rank_tc.cu): the in-order sum of a split tile's fp32 partials, batched
// transposes with zero padding (rank sides as K-major operands), and
// zero-padded copies of rank-r matrices whose rank is not a multiple of 8.
#include <algorithm>

#include "rank_store.cuh"

namespace lora {

namespace {

// Second pass: out = sum of a tile's unit partials, in unit order.  One
// thread per 4 consecutive elements of [tile][tile_rows][rpad] of every
// problem with several units (rpad is a multiple of 16, so the 4 share a
// row); the loads of all units are independent and issued together.
template <typename Batch, bool kRow>
__global__ void __launch_bounds__(256) reduce_partials_kernel(const __grid_constant__ Batch b, int total4) {
  griddep_wait();
  griddep_launch_dependents();
  const int i4 = blockIdx.x * blockDim.x + threadIdx.x;
  if (i4 >= total4) return;
  const int i = i4 * 4;
  int pi = 0;
  while (pi + 1 < b.n && i >= (int)b.p[pi + 1].red_begin) ++pi;
  const auto& P = b.p[pi];
  const int e = i - P.red_begin;
  const int rpad = P.rpad, upt = P.upt;
  const int blk = b.tile_rows * rpad;
  const int tile = e / blk, k = e % blk;
  const float4* src = reinterpret_cast<const float4*>(b.partials + P.part_off + (size_t)tile * upt * blk + k);
  const size_t stride4 = (size_t)blk / 4;
  float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
  for (int u = 0; u < upt; ++u) {
    const float4 w = __ldcg(src + (size_t)u * stride4);
    v.x += w.x;
    v.y += w.y;
    v.z += w.z;
    v.w += w.w;
  }
  const int row = tile * b.tile_rows + k / rpad, j = k % rpad;
  const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    if constexpr (kRow) {
      if (row < P.T) row_store(P, row, j + q, vv[q]);
    } else {
      if (row < P.C) col_store(P, row, j + q, vv[q]);
    }
  }
}

// Batched transposes with zero padding (the rank side of sv = s dy B as a
// K-major operand of the tensor cores): job blockIdx.y, output element
// (j, n) per thread, n fastest so that the writes coalesce.
__global__ void transposes_kernel(const __grid_constant__ TransposeJobs jobs) {
  griddep_wait();
  griddep_launch_dependents();
  const int k = blockIdx.y;
  const int n = jobs.n[k];
  const long long total = (long long)n * jobs.r8[k];
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int j = (int)(e / n);
    const long long c = e % n;
    jobs.dst[k][e] = j < jobs.r[k] ? jobs.src[k][c * jobs.ld[k] + j] : __float2bfloat16_rn(0.f);
  }
}

__global__ void pad_cols_kernel(const __nv_bfloat16* __restrict__ src, int rows, int r,
                                __nv_bfloat16* __restrict__ dst, int ld_dst) {
  griddep_wait();
  griddep_launch_dependents();
  const size_t n = (size_t)rows * ld_dst;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const size_t row = i / ld_dst;
    const int j = (int)(i % ld_dst);
    dst[i] = j < r ? src[row * r + j] : __float2bfloat16_rn(0.f);
  }
}

// Failure-detection self-check: one thread waits, with the library's bounded
// wait, on a barrier that nothing arrives on; the wait gives up after
// limit_ns, records the timeout in the status word and the kernel returns.
__global__ void wait_probe_kernel(int* status, long long limit_ns) {
  griddep_wait();
  griddep_launch_dependents();
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    abort_flag = 0;
    fence_mbar_init();
    const WaitCtl wc{status, limit_ns};
    mbar_wait(smem_u32(&bar), 0, wc, &abort_flag);
  }
}

int grid_for(size_t n, int threads) {
  size_t b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 65535) b = 65535;
  return (int)b;
}

}  // namespace

cudaError_t launch_transposes(const TransposeJobs& jobs, cudaStream_t st) {
  if (jobs.count <= 0 || jobs.max_elems <= 0) return cudaSuccess;
  const int bx = std::min(grid_for((size_t)jobs.max_elems, 256), 64);
  return launch_kernel(transposes_kernel, dim3(bx, jobs.count), dim3(256), 0, st, 1, jobs);
}

cudaError_t launch_reduce_rows(const RowBatch& b, cudaStream_t st) {
  if (b.red_total <= 0) return cudaSuccess;
  const int total4 = b.red_total / 4;
  return launch_kernel(reduce_partials_kernel<RowBatch, true>, dim3((total4 + 255) / 256), dim3(256), 0, st, 1, b,
                       total4);
}

cudaError_t launch_wait_probe(int* status, long long limit_ns, cudaStream_t st) {
  return launch_kernel(wait_probe_kernel, dim3(1), dim3(32), 0, st, 1, status, limit_ns);
}

cudaError_t launch_reduce_cols(const ColBatch& b, cudaStream_t st) {
  if (b.red_total <= 0) return cudaSuccess;
  const int total4 = b.red_total / 4;
  return launch_kernel(reduce_partials_kernel<ColBatch, false>, dim3((total4 + 255) / 256), dim3(256), 0, st, 1, b,
                       total4);
}

cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t st) {
  const size_t n = (size_t)rows * ld_dst;
  return launch_kernel(pad_cols_kernel, dim3(grid_for(n, 256)), dim3(256), 0, st, 1, src, rows, r, dst, ld_dst);
}

}  // namespace lora
