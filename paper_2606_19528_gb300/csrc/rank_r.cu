// Bandwidth-bound rank-r products of the LoRA linear:
//   su = s x A^T   and   sv = s dy B          (row products, reduce over columns)
//   dB = dy^T su   and   dA = sv^T x          (column products, reduce over tokens)
// Each reads one tall [T, C] bf16 activation once; the rank-r side is small
// and stays in L2.  Tiles of 64 x 64 are staged in shared memory with
// 16-byte cp.async copies (two-stage ring), fed to the legacy warp-level
// bf16 MMA (m16n8k16, fp32 accumulate) through ldmatrix, because at r >= 16
// the FMA pipes cannot keep up with HBM.  Reductions that are split across
// CTAs write fp32 partials that a second pass sums in a fixed order, so
// results do not depend on scheduling.
#include "common.cuh"
#include "kernels.h"

namespace lora {

namespace {

constexpr int kTile = 64;        // tokens x columns per tile
constexpr int kXPitch = 72;      // padded row of the X tile (bf16), 144 B: conflict-free ldmatrix
constexpr int kThreads = 128;    // 4 warps

template <int R>
struct RankTile {
  // W tile of a row product in [R, 64] (w_rc) or [64, R] form; S tile of a column product [64, R].
  static constexpr int kRcPitch = kXPitch;  // [R][72]
  static constexpr int kCrPitch = R + 8;    // [64][R + 8]
  static constexpr int kXBytes = kTile * kXPitch * 2;
  static constexpr int kWBytesRc = R * kRcPitch * 2;
  static constexpr int kWBytesCr = kTile * kCrPitch * 2;
  static constexpr int kWBytes = kWBytesRc > kWBytesCr ? kWBytesRc : kWBytesCr;
  static constexpr int kStageBytes = kXBytes + kWBytes;
  static constexpr int kSmem = 2 * kStageBytes;
};

// ----------------------------------------------------------------- row product
template <int R, bool kWRc>
__global__ void __launch_bounds__(kThreads) rowproj_kernel(const __nv_bfloat16* __restrict__ X, int ldx,
                                                           const __nv_bfloat16* __restrict__ Wm, int ldw,
                                                           int T, int C, int r, int chunks_per_split,
                                                           float* __restrict__ part,
                                                           __nv_bfloat16* __restrict__ out, int ld_out,
                                                           __nv_bfloat16* __restrict__ out2, int ld_out2,
                                                           float scale) {
  using L = RankTile<R>;
  constexpr int NT = R / 8;
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t0 = blockIdx.x * kTile;
  const int c_begin = blockIdx.y * chunks_per_split * kTile;
  const int c_end = min(C, c_begin + chunks_per_split * kTile);
  const int nch = (c_end - c_begin + kTile - 1) / kTile;

  auto load = [&](int s, int ch) {
    const uint32_t xs = sbase + s * L::kStageBytes;
    const uint32_t ws = xs + L::kXBytes;
    const int c0 = c_begin + ch * kTile;
    for (int i = threadIdx.x; i < kTile * 8; i += kThreads) {
      const int row = i >> 3, cc = (i & 7) * 8;
      const bool ok = (t0 + row < T) && (c0 + cc < c_end);
      const __nv_bfloat16* src = ok ? X + (size_t)(t0 + row) * ldx + c0 + cc : X;
      cp_async_16(xs + (row * kXPitch + cc) * 2, src, ok ? 16u : 0u);
    }
    if (kWRc) {
      for (int i = threadIdx.x; i < R * 8; i += kThreads) {
        const int j = i >> 3, cc = (i & 7) * 8;
        const bool ok = (j < r) && (c0 + cc < c_end);
        const __nv_bfloat16* src = ok ? Wm + (size_t)j * ldw + c0 + cc : Wm;
        cp_async_16(ws + (j * L::kRcPitch + cc) * 2, src, ok ? 16u : 0u);
      }
    } else {
      constexpr int JC = R / 8;
      for (int i = threadIdx.x; i < kTile * JC; i += kThreads) {
        const int c = i / JC, jj = (i % JC) * 8;
        const bool ok = (c0 + c < c_end) && (jj < ldw);
        const __nv_bfloat16* src = ok ? Wm + (size_t)(c0 + c) * ldw + jj : Wm;
        cp_async_16(ws + (c * L::kCrPitch + jj) * 2, src, ok ? 16u : 0u);
      }
    }
    cp_async_commit();
  };

  float acc[NT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;

  if (nch > 0) load(0, 0);
  for (int ch = 0; ch < nch; ++ch) {
    if (ch + 1 < nch)
      load((ch + 1) & 1, ch + 1);
    else
      cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    const uint32_t xs = sbase + (ch & 1) * L::kStageBytes;
    const uint32_t ws = xs + L::kXBytes;
    const int mi = lane >> 3, rr = lane & 7;
#pragma unroll
    for (int ks = 0; ks < kTile / 16; ++ks) {
      uint32_t a0, a1, a2, a3;
      ldsm_x4(xs + ((warp * 16 + (lane & 15)) * kXPitch + ks * 16 + (lane >> 4) * 8) * 2, a0, a1, a2, a3);
#pragma unroll
      for (int n = 0; n < NT; n += 2) {
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
    __syncthreads();
  }

  const int g = lane >> 2, q = lane & 3;
#pragma unroll
  for (int n = 0; n < NT; ++n) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int t = t0 + warp * 16 + g + h * 8;
      if (t >= T) continue;
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = n * 8 + 2 * q + e;
        const float v = acc[n][h * 2 + e];
        if (gridDim.y == 1) {
          const __nv_bfloat16 o = __float2bfloat16_rn(scale * v);
          if (j < ld_out) out[(size_t)t * ld_out + j] = j < r ? o : __float2bfloat16_rn(0.f);
          if (out2 != nullptr && j < ld_out2) out2[(size_t)t * ld_out2 + j] = j < r ? o : __float2bfloat16_rn(0.f);
        } else if (j < r) {
          part[((size_t)blockIdx.y * T + t) * r + j] = v;
        }
      }
    }
  }
}

// Finishes a split row product: out[t, j] = bf16(scale * sum_s part[s, t, j]).
__global__ void reduce_rows_kernel(const float* __restrict__ part, int splits, int T, int r,
                                   __nv_bfloat16* __restrict__ out, int ld_out,
                                   __nv_bfloat16* __restrict__ out2, int ld_out2, float scale) {
  const int ld = ld_out > ld_out2 ? ld_out : ld_out2;
  const size_t n = (size_t)T * ld;
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    const int t = (int)(i / ld), j = (int)(i % ld);
    float s = 0.f;
    if (j < r)
      for (int k = 0; k < splits; ++k) s += part[((size_t)k * T + t) * r + j];
    const __nv_bfloat16 o = __float2bfloat16_rn(scale * s);
    if (j < ld_out) out[(size_t)t * ld_out + j] = o;
    if (out2 != nullptr && j < ld_out2) out2[(size_t)t * ld_out2 + j] = o;
  }
}

// ----------------------------------------------------------------- column product
template <int R, bool kOutCr>
__global__ void __launch_bounds__(kThreads) colproj_kernel(const __nv_bfloat16* __restrict__ X, int ldx,
                                                           const __nv_bfloat16* __restrict__ S, int lds,
                                                           int T, int C, int r, int chunks_per_split,
                                                           float* __restrict__ part, float* __restrict__ out) {
  using L = RankTile<R>;
  constexpr int NT = R / 8;
  extern __shared__ __align__(16) uint8_t smem[];
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c0 = blockIdx.x * kTile;
  const int t_begin = blockIdx.y * chunks_per_split * kTile;
  const int t_end = min(T, t_begin + chunks_per_split * kTile);
  const int nch = (t_end - t_begin + kTile - 1) / kTile;

  auto load = [&](int s, int ch) {
    const uint32_t xs = sbase + s * L::kStageBytes;
    const uint32_t ss = xs + L::kXBytes;
    const int tb = t_begin + ch * kTile;
    for (int i = threadIdx.x; i < kTile * 8; i += kThreads) {
      const int row = i >> 3, cc = (i & 7) * 8;
      const bool ok = (tb + row < t_end) && (c0 + cc < C);
      const __nv_bfloat16* src = ok ? X + (size_t)(tb + row) * ldx + c0 + cc : X;
      cp_async_16(xs + (row * kXPitch + cc) * 2, src, ok ? 16u : 0u);
    }
    constexpr int JC = R / 8;
    for (int i = threadIdx.x; i < kTile * JC; i += kThreads) {
      const int row = i / JC, jj = (i % JC) * 8;
      const bool ok = (tb + row < t_end) && (jj < lds);
      const __nv_bfloat16* src = ok ? S + (size_t)(tb + row) * lds + jj : S;
      cp_async_16(ss + (row * L::kCrPitch + jj) * 2, src, ok ? 16u : 0u);
    }
    cp_async_commit();
  };

  float acc[NT][4];
#pragma unroll
  for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;

  if (nch > 0) load(0, 0);
  for (int ch = 0; ch < nch; ++ch) {
    if (ch + 1 < nch)
      load((ch + 1) & 1, ch + 1);
    else
      cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    const uint32_t xs = sbase + (ch & 1) * L::kStageBytes;
    const uint32_t ss = xs + L::kXBytes;
    const int mi = lane >> 3, rr = lane & 7;
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
        uint32_t b0, b1, b2, b3;
        const int t = ks * 16 + (mi & 1) * 8 + rr;
        const int j = (n + (mi >> 1)) * 8;
        ldsm_x4_t(ss + (t * L::kCrPitch + j) * 2, b0, b1, b2, b3);
        mma_16816(acc[n], a0, a1, a2, a3, b0, b1);
        mma_16816(acc[n + 1], a0, a1, a2, a3, b2, b3);
      }
    }
    __syncthreads();
  }

  const int g = lane >> 2, q = lane & 3;
  float* dst = gridDim.y == 1 ? out : part + (size_t)blockIdx.y * C * r;
#pragma unroll
  for (int n = 0; n < NT; ++n) {
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int c = c0 + warp * 16 + g + h * 8;
      if (c >= C) continue;
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = n * 8 + 2 * q + e;
        if (j >= r) continue;
        const float v = acc[n][h * 2 + e];
        if (kOutCr)
          dst[(size_t)c * r + j] = v;
        else
          dst[(size_t)j * C + c] = v;
      }
    }
  }
}

// out[i] = sum_s part[s * n + i] in fixed order.
__global__ void reduce_flat_kernel(const float* __restrict__ part, int splits, size_t n, float* __restrict__ out) {
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += part[(size_t)k * n + i];
    out[i] = s;
  }
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

int grid_for(size_t n, int threads) {
  size_t b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 65535) b = 65535;
  return (int)b;
}

// Raises the dynamic shared-memory limit of `kernel` once per process.
template <typename K>
cudaError_t set_smem(K kernel, int bytes) {
  static bool done = false;  // one flag per kernel instantiation
  if (done) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess) done = true;
  return e;
}

template <int R>
cudaError_t rowproj_r(const __nv_bfloat16* X, int ldx, const __nv_bfloat16* Wm, int ldw, bool w_rc, int T,
                      int C, int r, const RowProjPlan& plan, float* part, __nv_bfloat16* out, int ld_out,
                      __nv_bfloat16* out2, int ld_out2, float scale, cudaStream_t st) {
  constexpr int smem = RankTile<R>::kSmem;
  dim3 grid((T + kTile - 1) / kTile, plan.splits);
  cudaError_t e;
  if (w_rc) {
    if ((e = set_smem(rowproj_kernel<R, true>, smem)) != cudaSuccess) return e;
    rowproj_kernel<R, true><<<grid, kThreads, smem, st>>>(X, ldx, Wm, ldw, T, C, r, plan.chunks_per_split, part,
                                                          out, ld_out, out2, ld_out2, scale);
    note_launch();
  } else {
    if ((e = set_smem(rowproj_kernel<R, false>, smem)) != cudaSuccess) return e;
    rowproj_kernel<R, false><<<grid, kThreads, smem, st>>>(X, ldx, Wm, ldw, T, C, r, plan.chunks_per_split, part,
                                                           out, ld_out, out2, ld_out2, scale);
    note_launch();
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (plan.splits > 1) {
    const int ld = ld_out > ld_out2 ? ld_out : ld_out2;
    reduce_rows_kernel<<<grid_for((size_t)T * ld, 256), 256, 0, st>>>(part, plan.splits, T, r, out, ld_out, out2,
                                                                        ld_out2, scale);
    note_launch();
    e = cudaGetLastError();
  }
  return e;
}

template <int R>
cudaError_t colproj_r(const __nv_bfloat16* X, int ldx, const __nv_bfloat16* S, int lds, int T, int C, int r,
                      const ColProjPlan& plan, float* part, float* out, bool out_cr, cudaStream_t st) {
  constexpr int smem = RankTile<R>::kSmem;
  dim3 grid((C + kTile - 1) / kTile, plan.splits);
  cudaError_t e;
  if (out_cr) {
    if ((e = set_smem(colproj_kernel<R, true>, smem)) != cudaSuccess) return e;
    colproj_kernel<R, true><<<grid, kThreads, smem, st>>>(X, ldx, S, lds, T, C, r, plan.chunks_per_split, part, out);
    note_launch();
  } else {
    if ((e = set_smem(colproj_kernel<R, false>, smem)) != cudaSuccess) return e;
    colproj_kernel<R, false><<<grid, kThreads, smem, st>>>(X, ldx, S, lds, T, C, r, plan.chunks_per_split, part, out);
    note_launch();
  }
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (plan.splits > 1) {
    const size_t n = (size_t)C * r;
    reduce_flat_kernel<<<grid_for(n, 256), 256, 0, st>>>(part, plan.splits, n, out);
    note_launch();
    e = cudaGetLastError();
  }
  return e;
}

}  // namespace

static int split_count(int tiles, int chunks, int num_sms, int* per_split) {
  const int target = 4 * num_sms;
  int splits = (target + tiles - 1) / tiles;
  if (splits < 1) splits = 1;
  if (splits > chunks) splits = chunks;
  if (splits > 32) splits = 32;
  const int cps = (chunks + splits - 1) / splits;
  *per_split = cps;
  return (chunks + cps - 1) / cps;
}

RowProjPlan plan_rowproj(int T, int C, int num_sms) {
  RowProjPlan p;
  const int chunks = (C + kTile - 1) / kTile;
  p.splits = split_count((T + kTile - 1) / kTile, chunks, num_sms, &p.chunks_per_split);
  return p;
}

ColProjPlan plan_colproj(int T, int C, int num_sms) {
  ColProjPlan p;
  const int chunks = (T + kTile - 1) / kTile;
  p.splits = split_count((C + kTile - 1) / kTile, chunks, num_sms, &p.chunks_per_split);
  return p;
}

cudaError_t launch_rowproj(const __nv_bfloat16* X, int ldx, const __nv_bfloat16* Wm, int ldw, bool w_rc, int T,
                           int C, int r, const RowProjPlan& plan, float* part, __nv_bfloat16* out, int ld_out,
                           __nv_bfloat16* out2, int ld_out2, float scale, cudaStream_t st) {
  const int R = rank_pad16(r);
  switch (R) {
    case 16: return rowproj_r<16>(X, ldx, Wm, ldw, w_rc, T, C, r, plan, part, out, ld_out, out2, ld_out2, scale, st);
    case 32: return rowproj_r<32>(X, ldx, Wm, ldw, w_rc, T, C, r, plan, part, out, ld_out, out2, ld_out2, scale, st);
    case 48:
    case 64: return rowproj_r<64>(X, ldx, Wm, ldw, w_rc, T, C, r, plan, part, out, ld_out, out2, ld_out2, scale, st);
    default: return rowproj_r<128>(X, ldx, Wm, ldw, w_rc, T, C, r, plan, part, out, ld_out, out2, ld_out2, scale, st);
  }
}

cudaError_t launch_colproj(const __nv_bfloat16* X, int ldx, const __nv_bfloat16* S, int lds, int T, int C, int r,
                           const ColProjPlan& plan, float* part, float* out, bool out_cr, cudaStream_t st) {
  const int R = rank_pad16(r);
  switch (R) {
    case 16: return colproj_r<16>(X, ldx, S, lds, T, C, r, plan, part, out, out_cr, st);
    case 32: return colproj_r<32>(X, ldx, S, lds, T, C, r, plan, part, out, out_cr, st);
    case 48:
    case 64: return colproj_r<64>(X, ldx, S, lds, T, C, r, plan, part, out, out_cr, st);
    default: return colproj_r<128>(X, ldx, S, lds, T, C, r, plan, part, out, out_cr, st);
  }
}

cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t st) {
  const size_t n = (size_t)rows * ld_dst;
  pad_cols_kernel<<<grid_for(n, 256), 256, 0, st>>>(src, rows, r, dst, ld_dst);
  note_launch();
  return cudaGetLastError();
}

}  // namespace lora
