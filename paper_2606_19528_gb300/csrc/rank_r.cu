// Bandwidth-bound rank-r products of the LoRA linear:
//   row products     su = s x A^T,  sv = s dy B      out[t, j], reduced over columns c
//   column products  dB = dy^T su,  dA = sv^T x      out[c, j], reduced over tokens t
// Each problem streams one tall [T, C] bf16 activation X once; the rank side
// (A, B, su or sv) is small and stays in L2.  Projections that read the same
// X are one problem whose rank side is the concatenation of theirs (q, k and
// v read x once for all three).  One launch covers every problem of a phase.
//
// Tiles of 64 x 64 of X are staged in shared memory by 16-byte cp.async
// copies through a three-stage ring and fed to the warp-level bf16 MMA
// (m16n8k16, fp32 accumulate) through ldmatrix; at r >= 16 FMA pipes could
// not keep up with HBM.  When a problem has too few tiles to fill the GPU,
// its reduction is split across the CTAs of a thread-block cluster (up to
// 8); their fp32 partials are summed through distributed shared memory in
// cluster-rank order, so results never depend on scheduling.
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

namespace lora {

namespace {

constexpr int kTile = 64;      // tokens x columns per tile
constexpr int kXPitch = 72;    // padded X-tile row (bf16): 144 B keeps ldmatrix conflict-free
constexpr int kThreads = 128;  // 4 warps, 16 rows (row product) or 16 columns (column product) each
constexpr int kStages = 3;

template <int R>
struct Smem {
  static constexpr int kRcPitch = kXPitch;  // rank-side tile [R][72] (row product with A)
  static constexpr int kCrPitch = R + 8;    // rank-side tile [64][R + 8]
  static constexpr int kXBytes = kTile * kXPitch * 2;
  static constexpr int kWBytes = (R * kRcPitch > kTile * kCrPitch ? R * kRcPitch : kTile * kCrPitch) * 2;
  static constexpr int kStageBytes = kXBytes + kWBytes;
  static constexpr int kPartPitch = R + 4;  // fp32 partial tile [64][R + 4]
  static constexpr int kPartBytes = kTile * kPartPitch * 4;
  static constexpr int kBytes =
      kStages * kStageBytes > kPartBytes ? kStages * kStageBytes : kPartBytes;
};

__device__ __forceinline__ int pad8(int r) { return (r + 7) & ~7; }

// Block of concatenated rank column j (blocks are packed at 8-aligned offsets).
__device__ __forceinline__ int find_block(const int* rw, int nblk, int j, int* jj) {
  int off = 0;
  for (int b = 0; b < nblk; ++b) {
    const int w = pad8(rw[b]);
    if (j < off + w) {
      *jj = j - off;
      return b;
    }
    off += w;
  }
  return -1;
}

__device__ __forceinline__ void row_store(const RowProb& P, int t, int j, float v) {
  int jj;
  const int b = find_block(P.rw, P.nblk, j, &jj);
  if (b < 0) return;
  const __nv_bfloat16 o = __float2bfloat16_rn(jj < P.rw[b] ? P.scale * v : 0.f);
  if (jj < P.ld_out[b]) P.out[b][(size_t)t * P.ld_out[b] + jj] = o;
  if (P.out2[b] != nullptr && jj < P.ld_out2[b]) P.out2[b][(size_t)t * P.ld_out2[b] + jj] = o;
}

__device__ __forceinline__ void col_store(const ColProb& P, int c, int j, float v) {
  int jj;
  const int b = find_block(P.rs, P.nblk, j, &jj);
  if (b < 0 || jj >= P.rs[b]) return;
  if (P.out_cr)
    P.out[b][(size_t)c * P.rs[b] + jj] = v;
  else
    P.out[b][(size_t)jj * P.C + c] = v;
}

// Writes the warp's 16 x rpad accumulator tile into the fp32 partial tile.
template <int R>
__device__ __forceinline__ void acc_to_smem(float* part, const float (&acc)[R / 8][4], int warp, int lane, int ntp) {
  const int g = lane >> 2, q = lane & 3;
#pragma unroll
  for (int n = 0; n < R / 8; ++n) {
    if (n < ntp) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float* row = part + (warp * 16 + g + h * 8) * Smem<R>::kPartPitch + n * 8 + 2 * q;
        row[0] = acc[n][h * 2];
        row[1] = acc[n][h * 2 + 1];
      }
    }
  }
}

// ------------------------------------------------------------------------- row products
template <int R, bool kWRc>
__global__ void __launch_bounds__(kThreads) rowprod_kernel(const __grid_constant__ RowBatch b) {
  using L = Smem<R>;
  constexpr int NT = R / 8;
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  int pi = 0;
  while (pi + 1 < b.n && (int)blockIdx.x >= b.p[pi + 1].tile_begin) ++pi;
  const RowProb& P = b.p[pi];
  const int t0 = ((int)blockIdx.x - P.tile_begin) * kTile;
  const int c_begin = blockIdx.y * P.cps * kTile;
  const int c_end = min(P.C, c_begin + P.cps * kTile);
  const int nch = c_end > c_begin ? (c_end - c_begin + kTile - 1) / kTile : 0;
  const int ntp = P.rpad / 8;

  auto load = [&](int s, int ch) {
    const uint32_t xs = sbase + s * L::kStageBytes;
    const uint32_t ws = xs + L::kXBytes;
    const int c0 = c_begin + ch * kTile;
    for (int i = threadIdx.x; i < kTile * 8; i += kThreads) {
      const int row = i >> 3, cc = (i & 7) * 8;
      const bool ok = (t0 + row < P.T) && (c0 + cc < c_end);
      const __nv_bfloat16* src = ok ? P.X + (size_t)(t0 + row) * P.ldx + c0 + cc : P.X;
      cp_async_16(xs + (row * kXPitch + cc) * 2, src, ok ? 16u : 0u);
    }
    if (kWRc) {
      // rank rows j of the concatenated [A_0; A_1; ...], each block 8-row aligned
      for (int i = threadIdx.x; i < P.rpad * 8; i += kThreads) {
        const int j = i >> 3, cc = (i & 7) * 8;
        int jj;
        const int bb = find_block(P.rw, P.nblk, j, &jj);
        const bool ok = bb >= 0 && jj < P.rw[bb] && (c0 + cc < c_end);
        const __nv_bfloat16* src = ok ? P.W[bb] + (size_t)jj * P.ldw[bb] + c0 + cc : P.X;
        cp_async_16(ws + (j * L::kRcPitch + cc) * 2, src, ok ? 16u : 0u);
      }
    } else {
      // B [C, r] of one projection, row stride ldw[0] (a multiple of 8)
      const int jc = P.rpad / 8;
      for (int i = threadIdx.x; i < kTile * jc; i += kThreads) {
        const int c = i / jc, jj = (i % jc) * 8;
        const bool ok = (c0 + c < c_end) && (jj < P.ldw[0]);
        const __nv_bfloat16* src = ok ? P.W[0] + (size_t)(c0 + c) * P.ldw[0] + jj : P.X;
        cp_async_16(ws + (c * L::kCrPitch + jj) * 2, src, ok ? 16u : 0u);
      }
    }
  };

  float acc[NT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;

#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    if (s < nch) load(s, s);
    cp_async_commit();
  }
  const int mi = lane >> 3, rr = lane & 7;
  for (int ch = 0; ch < nch; ++ch) {
    cp_async_wait<kStages - 2>();
    __syncthreads();
    if (ch + kStages - 1 < nch) load((ch + kStages - 1) % kStages, ch + kStages - 1);
    cp_async_commit();
    const uint32_t xs = sbase + (ch % kStages) * L::kStageBytes;
    const uint32_t ws = xs + L::kXBytes;
#pragma unroll
    for (int ks = 0; ks < kTile / 16; ++ks) {
      uint32_t a0, a1, a2, a3;
      ldsm_x4(xs + ((warp * 16 + (lane & 15)) * kXPitch + ks * 16 + (lane >> 4) * 8) * 2, a0, a1, a2, a3);
#pragma unroll
      for (int n = 0; n < NT; n += 2) {
        if (n < ntp) {
          uint32_t b0, b1, b2, b3;
          if (kWRc) {
            const int j = (n + (mi >> 1)) * 8 + rr;
            const int c = ks * 16 + (mi & 1) * 8;
            ldsm_x4(ws + (j * L::kRcPitch + c) * 2, b0, b1, b2, b3);
          } else {
            const int c = ks * 16 + (mi & 1) * 8 + rr;
            const int j = (n + (mi >> 1)) * 8;
            ldsm_x4_t(ws + (c * L::kCrPitch + j) * 2, b0, b1, b2, b3);
          }
          mma_16816(acc[n], a0, a1, a2, a3, b0, b1);
          mma_16816(acc[n + 1], a0, a1, a2, a3, b2, b3);
        }
      }
    }
  }
  cp_async_wait<0>();
  __syncthreads();

  if (gridDim.y == 1) {
    const int g = lane >> 2, q = lane & 3;
#pragma unroll
    for (int n = 0; n < NT; ++n) {
      if (n < ntp) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int t = t0 + warp * 16 + g + h * 8;
          if (t < P.T) {
            row_store(P, t, n * 8 + 2 * q, acc[n][h * 2]);
            row_store(P, t, n * 8 + 2 * q + 1, acc[n][h * 2 + 1]);
          }
        }
      }
    }
    return;
  }

  // split reduction across the cluster: CTA of rank s sums rows [s*64/S, (s+1)*64/S)
  cg::cluster_group cluster = cg::this_cluster();
  float* part = reinterpret_cast<float*>(smem);
  acc_to_smem<R>(part, acc, warp, lane, ntp);
  cluster.sync();
  const int S = (int)gridDim.y;
  const int rows = kTile / S;
  const int r0 = (int)cluster.block_rank() * rows;
  for (int i = threadIdx.x; i < rows * P.rpad; i += kThreads) {
    const int row = r0 + i / P.rpad, j = i % P.rpad;
    float v = 0.f;
    for (int s = 0; s < S; ++s) v += cluster.map_shared_rank(part, s)[row * L::kPartPitch + j];
    const int t = t0 + row;
    if (t < P.T) row_store(P, t, j, v);
  }
  cluster.sync();
}

// ------------------------------------------------------------------------- column products
template <int R>
__global__ void __launch_bounds__(kThreads) colprod_kernel(const __grid_constant__ ColBatch b) {
  using L = Smem<R>;
  constexpr int NT = R / 8;
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  int pi = 0;
  while (pi + 1 < b.n && (int)blockIdx.x >= b.p[pi + 1].tile_begin) ++pi;
  const ColProb& P = b.p[pi];
  const int c0 = ((int)blockIdx.x - P.tile_begin) * kTile;
  const int t_begin = blockIdx.y * P.cps * kTile;
  const int t_end = min(P.T, t_begin + P.cps * kTile);
  const int nch = t_end > t_begin ? (t_end - t_begin + kTile - 1) / kTile : 0;
  const int ntp = P.rpad / 8;

  auto load = [&](int s, int ch) {
    const uint32_t xs = sbase + s * L::kStageBytes;
    const uint32_t ss = xs + L::kXBytes;
    const int tb = t_begin + ch * kTile;
    for (int i = threadIdx.x; i < kTile * 8; i += kThreads) {
      const int row = i >> 3, cc = (i & 7) * 8;
      const bool ok = (tb + row < t_end) && (c0 + cc < P.C);
      const __nv_bfloat16* src = ok ? P.X + (size_t)(tb + row) * P.ldx + c0 + cc : P.X;
      cp_async_16(xs + (row * kXPitch + cc) * 2, src, ok ? 16u : 0u);
    }
    // concatenated rank side [S_0 | S_1 | ...], blocks at 8-aligned columns
    const int jc = P.rpad / 8;
    for (int i = threadIdx.x; i < kTile * jc; i += kThreads) {
      const int row = i / jc, j = (i % jc) * 8;
      int jj;
      const int bb = find_block(P.rs, P.nblk, j, &jj);
      const bool ok = bb >= 0 && (tb + row < t_end) && (jj < P.lds[bb]);
      const __nv_bfloat16* src = ok ? P.S[bb] + (size_t)(tb + row) * P.lds[bb] + jj : P.X;
      cp_async_16(ss + (row * L::kCrPitch + j) * 2, src, ok ? 16u : 0u);
    }
  };

  float acc[NT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;

#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    if (s < nch) load(s, s);
    cp_async_commit();
  }
  const int mi = lane >> 3, rr = lane & 7;
  for (int ch = 0; ch < nch; ++ch) {
    cp_async_wait<kStages - 2>();
    __syncthreads();
    if (ch + kStages - 1 < nch) load((ch + kStages - 1) % kStages, ch + kStages - 1);
    cp_async_commit();
    const uint32_t xs = sbase + (ch % kStages) * L::kStageBytes;
    const uint32_t ss = xs + L::kXBytes;
#pragma unroll
    for (int ks = 0; ks < kTile / 16; ++ks) {
      // A(m = column c, k = token t) = X[t, c]: the staged tile is k-major, so load transposed
      uint32_t a0, a1, a2, a3;
      {
        const int t = ks * 16 + (mi >> 1) * 8 + rr;
        const int c = warp * 16 + (mi & 1) * 8;
        ldsm_x4_t(xs + (t * kXPitch + c) * 2, a0, a1, a2, a3);
      }
#pragma unroll
      for (int n = 0; n < NT; n += 2) {
        if (n < ntp) {
          uint32_t b0, b1, b2, b3;
          const int t = ks * 16 + (mi & 1) * 8 + rr;
          const int j = (n + (mi >> 1)) * 8;
          ldsm_x4_t(ss + (t * L::kCrPitch + j) * 2, b0, b1, b2, b3);
          mma_16816(acc[n], a0, a1, a2, a3, b0, b1);
          mma_16816(acc[n + 1], a0, a1, a2, a3, b2, b3);
        }
      }
    }
  }
  cp_async_wait<0>();
  __syncthreads();

  if (gridDim.y == 1) {
    const int g = lane >> 2, q = lane & 3;
#pragma unroll
    for (int n = 0; n < NT; ++n) {
      if (n < ntp) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int c = c0 + warp * 16 + g + h * 8;
          if (c < P.C) {
            col_store(P, c, n * 8 + 2 * q, acc[n][h * 2]);
            col_store(P, c, n * 8 + 2 * q + 1, acc[n][h * 2 + 1]);
          }
        }
      }
    }
    return;
  }

  cg::cluster_group cluster = cg::this_cluster();
  float* part = reinterpret_cast<float*>(smem);
  acc_to_smem<R>(part, acc, warp, lane, ntp);
  cluster.sync();
  const int S = (int)gridDim.y;
  const int rows = kTile / S;
  const int r0 = (int)cluster.block_rank() * rows;
  for (int i = threadIdx.x; i < rows * P.rpad; i += kThreads) {
    const int row = r0 + i / P.rpad, j = i % P.rpad;
    float v = 0.f;
    for (int s = 0; s < S; ++s) v += cluster.map_shared_rank(part, s)[row * L::kPartPitch + j];
    const int c = c0 + row;
    if (c < P.C) col_store(P, c, j, v);
  }
  cluster.sync();
}

__global__ void pad_cols_kernel(const __nv_bfloat16* __restrict__ src, int rows, int r,
                                __nv_bfloat16* __restrict__ dst, int ld_dst) {
  const size_t n = (size_t)rows * ld_dst;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const size_t row = i / ld_dst;
    const int j = (int)(i % ld_dst);
    dst[i] = j < r ? src[row * r + j] : __float2bfloat16_rn(0.f);
  }
}

// Raises the dynamic shared-memory limit of one kernel instantiation once.
template <auto Kernel>
cudaError_t set_smem_once(int bytes) {
  static bool done = false;
  if (done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done = true;
  return e;
}

template <auto Kernel, typename Batch>
cudaError_t launch_cluster(const Batch& b, int tiles, int splits, int smem, cudaStream_t st) {
  cudaError_t e = set_smem_once<Kernel>(smem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)tiles, (unsigned)splits, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = (unsigned)splits;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, Kernel, b);
  note_launch();
  return e;
}

template <int R>
cudaError_t rowprod_r(const RowBatch& b, cudaStream_t st) {
  constexpr int smem = Smem<R>::kBytes;
  if (b.w_rc) return launch_cluster<rowprod_kernel<R, true>>(b, b.tiles, b.splits, smem, st);
  return launch_cluster<rowprod_kernel<R, false>>(b, b.tiles, b.splits, smem, st);
}

template <int R>
cudaError_t colprod_r(const ColBatch& b, cudaStream_t st) {
  constexpr int smem = Smem<R>::kBytes;
  return launch_cluster<colprod_kernel<R>>(b, b.tiles, b.splits, smem, st);
}

int grid_for(size_t n, int threads) {
  size_t b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 65535) b = 65535;
  return (int)b;
}

}  // namespace

int rank_splits(int tiles, int max_chunks, int num_sms) {
  int s = 1;
  while (s < 8 && tiles * s < 2 * num_sms && s * 2 <= max_chunks) s *= 2;
  return s;
}

int rank_tile() { return kTile; }

cudaError_t launch_rowprod(const RowBatch& b, int rmax, cudaStream_t st) {
  if (b.n <= 0 || b.tiles <= 0) return cudaSuccess;
  if (rmax <= 16) return rowprod_r<16>(b, st);
  if (rmax <= 32) return rowprod_r<32>(b, st);
  if (rmax <= 64) return rowprod_r<64>(b, st);
  return rowprod_r<128>(b, st);
}

cudaError_t launch_colprod(const ColBatch& b, int rmax, cudaStream_t st) {
  if (b.n <= 0 || b.tiles <= 0) return cudaSuccess;
  if (rmax <= 16) return colprod_r<16>(b, st);
  if (rmax <= 32) return colprod_r<32>(b, st);
  if (rmax <= 64) return colprod_r<64>(b, st);
  return colprod_r<128>(b, st);
}

cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t st) {
  const size_t n = (size_t)rows * ld_dst;
  pad_cols_kernel<<<grid_for(n, 256), 256, 0, st>>>(src, rows, r, dst, ld_dst);
  note_launch();
  return cudaGetLastError();
}

}  // namespace lora
