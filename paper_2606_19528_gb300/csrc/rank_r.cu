// Bandwidth-bound rank-r products of the LoRA linear:
//   row products     su = s x A^T,  sv = s dy B      out[t, j], reduced over columns c
//   column products  dB = dy^T su,  dA = sv^T x      out[c, j], reduced over tokens t
// Each problem streams one tall [T, C] bf16 activation X once; the rank side
// (A, B, su or sv) is small and stays in L2.  Projections that read the same
// X are one problem whose rank side is the concatenation of theirs (q, k and
// v read x once for all three).  One launch covers every problem of a phase.
//
// Streaming structure (per CTA, two CTAs per SM, persistent): one producer
// warp issues TMA loads of 64 x 64 tiles of X (128-byte swizzle) and of the
// matching rank-side tiles (zero-filled past each block's rank) into a deep
// ring of shared-memory stages guarded by mbarriers; four consumer warps
// turn each stage into warp-level bf16 MMAs (m16n8k16, fp32 accumulate) fed
// by ldmatrix — at r >= 16 FMA pipes could not keep up with HBM.  Work is cut
// into equal units of `unit_chunks` 64-wide chunks of the reduction taken
// round-robin, so every SM streams the same amount whatever the problem
// sizes, and a unit's epilogue overlaps the next unit's loads.  A tile whose
// reduction spans several units gets one fp32 partial per unit; a second,
// fully parallel pass sums them in unit order, so results never depend on
// scheduling.
#include "common.cuh"
#include "kernels.h"

namespace lora {

namespace {

constexpr int kTile = 64;         // tokens x columns per chunk
constexpr int kConsumers = 4;     // consumer warps: 16 rows (row product) or 16 columns (column product) each
constexpr int kThreads = (kConsumers + 1) * 32;
constexpr uint32_t kXBytes = kTile * kTile * 2;  // one 64 x 64 bf16 tile of X, 8 KB
constexpr long long kDrainNs = 1000000000ll;

// Shared-memory plan for a padded rank R: each stage holds the X tile and a
// rank-side tile of R x 64 bf16 (128 R bytes, whatever its orientation).
template <int R>
struct Ring {
  static constexpr uint32_t kStageBytes = (kXBytes + 128u * R + 1023u) & ~1023u;
  static constexpr int kStages = R <= 16 ? 10 : R <= 32 ? 8 : R <= 64 ? 6 : 4;
  static constexpr uint32_t kBytes = 1024 + kStages * kStageBytes + 2 * kStages * 8 + 16;
};

__device__ __forceinline__ int pad8(int r) { return (r + 7) & ~7; }

// Block of concatenated rank column j (blocks are packed at 8-aligned offsets).
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

// Byte offset of element (row, col) in a 64-column bf16 tile stored with the
// 128-byte swizzle of TMA (16-byte chunk index XOR row mod 8).
__device__ __forceinline__ uint32_t sw128(int row, int col) {
  return (uint32_t)(row * 128 + ((((col >> 3) ^ (row & 7)) & 7) << 4) + (col & 7) * 2);
}

__device__ __forceinline__ void consumers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kConsumers * 32) : "memory"); }

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

// The warp's 16-row slice of the accumulator tile as fp32 partial [64][rpad].
template <int R>
__device__ __forceinline__ void acc_to_partial(float* part, int rpad, const float (&acc)[R / 8][4], int warp, int lane,
                                               int ntp) {
  const int g = lane >> 2, q = lane & 3;
#pragma unroll
  for (int n = 0; n < R / 8; ++n) {
    if (n < ntp) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float2* dst = reinterpret_cast<float2*>(part + (size_t)(warp * 16 + g + h * 8) * rpad + n * 8 + 2 * q);
        __stcg(dst, make_float2(acc[n][h * 2], acc[n][h * 2 + 1]));
      }
    }
  }
}

struct RingCtl {
  uint32_t full0, empty0;  // addresses of full[0], empty[0]
  volatile int* abort;
};

template <int R>
__device__ __forceinline__ RingCtl ring_init(uint8_t* smem_raw, uint32_t* base_out) {
  using G = Ring<R>;
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* ctl = smem_raw + (base - raw) + (size_t)G::kStages * G::kStageBytes;
  RingCtl rc;
  rc.full0 = smem_u32(ctl);
  rc.empty0 = rc.full0 + 8u * G::kStages;
  rc.abort = reinterpret_cast<volatile int*>(ctl + 16 * G::kStages);
  if (threadIdx.x == 0) {
    for (int s = 0; s < G::kStages; ++s) {
      mbar_init(rc.full0 + 8u * s, 1);
      mbar_init(rc.empty0 + 8u * s, kConsumers);
    }
    *rc.abort = 0;
    fence_mbar_init();
  }
  __syncthreads();
  *base_out = base;
  return rc;
}

// Producer epilogue after a wait gave up: let the copies it issued land.
template <int R>
__device__ __forceinline__ void ring_drain(const RingCtl& rc, long long issued) {
  using G = Ring<R>;
  const long long first = issued > G::kStages ? issued - G::kStages : 0;
  for (long long j = first; j < issued; ++j)
    mbar_wait_drain(rc.full0 + 8u * (uint32_t)(j % G::kStages), (uint32_t)((j / G::kStages) & 1), kDrainNs);
}

// ------------------------------------------------------------------------- row products
template <int R, bool kWRc>
__global__ void __launch_bounds__(kThreads) rowprod_kernel(const __grid_constant__ RowBatch b) {
  using G = Ring<R>;
  constexpr int NT = R / 8;
  extern __shared__ uint8_t smem_raw[];
  uint32_t base;
  const RingCtl rc = ring_init<R>(smem_raw, &base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{b.status, b.limit_ns};

  if (warp == kConsumers) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < b.units && ok; u += gridDim.x) {
        int pi = 0;
        while (pi + 1 < b.n && u >= b.p[pi + 1].unit_begin) ++pi;
        const RowProb& P = b.p[pi];
        const int lu = u - P.unit_begin;
        const int t0 = (lu / P.upt) * kTile;
        const int c_begin = (lu % P.upt) * b.unit_chunks * kTile;
        const int nch = (min(P.C, c_begin + b.unit_chunks * kTile) - c_begin + kTile - 1) / kTile;
        for (int ch = 0; ch < nch; ++ch) {
          const uint32_t empty = rc.empty0 + 8u * stage, full = rc.full0 + 8u * stage;
          if (!mbar_wait(empty, phase ^ 1u, wc, rc.abort)) {
            ok = false;
            break;
          }
          const uint32_t xs = base + (uint32_t)stage * G::kStageBytes;
          const int c0 = c_begin + ch * kTile;
          mbar_arrive_expect_tx(full, (uint32_t)P.tx_bytes);
          tma_load_2d(xs, &P.tmX, full, c0, t0);
          if (kWRc) {
            int off = 0;
            for (int k = 0; k < P.nblk; ++k) {
              tma_load_2d(xs + kXBytes + (uint32_t)off * 128u, &P.tmW[k], full, c0, 0);
              off += pad8(P.rw[k]);
            }
          } else {
            tma_load_2d(xs + kXBytes, &P.tmW[0], full, 0, c0);
          }
          ++issued;
          if (++stage == G::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (*rc.abort) ring_drain<R>(rc, issued);
    }
    return;
  }

  // ------------------------------------------------------------------ consumers
  const int mi = lane >> 3, rr = lane & 7;
  int stage = 0;
  uint32_t phase = 0;
  for (int u = blockIdx.x; u < b.units; u += gridDim.x) {
    int pi = 0;
    while (pi + 1 < b.n && u >= b.p[pi + 1].unit_begin) ++pi;
    const RowProb& P = b.p[pi];
    const int lu = u - P.unit_begin;
    const int tile = lu / P.upt, piece = lu % P.upt;
    const int t0 = tile * kTile;
    const int c_begin = piece * b.unit_chunks * kTile;
    const int nch = (min(P.C, c_begin + b.unit_chunks * kTile) - c_begin + kTile - 1) / kTile;
    const int ntp = P.rpad / 8;
    const int r8 = pad8(P.rw[0]);  // row pitch of the B tile (one block) in elements

    float acc[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;

    bool ok = true;
    for (int ch = 0; ch < nch; ++ch) {
      ok = mbar_wait(rc.full0 + 8u * stage, phase, wc, rc.abort);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      const uint32_t xs = base + (uint32_t)stage * G::kStageBytes;
      const uint32_t ws = xs + kXBytes;
#pragma unroll
      for (int ks = 0; ks < kTile / 16; ++ks) {
        uint32_t a0, a1, a2, a3;
        ldsm_x4(xs + sw128(warp * 16 + (lane & 15), ks * 16 + (lane >> 4) * 8), a0, a1, a2, a3);
#pragma unroll
        for (int n = 0; n < NT; n += 2) {
          if (n < ntp) {
            uint32_t b0, b1, b2, b3;
            if (kWRc) {
              // A tile: rank rows j x 64 columns, 128-byte swizzle
              ldsm_x4(ws + sw128((n + (mi >> 1)) * 8 + rr, ks * 16 + (mi & 1) * 8), b0, b1, b2, b3);
            } else {
              // B tile: 64 column rows x r8 rank entries, dense
              const int c = ks * 16 + (mi & 1) * 8 + rr;
              const int j = (n + (mi >> 1)) * 8;
              ldsm_x4_t(ws + (uint32_t)(c * r8 + j) * 2u, b0, b1, b2, b3);
            }
            mma_16816(acc[n], a0, a1, a2, a3, b0, b1);
            mma_16816(acc[n + 1], a0, a1, a2, a3, b2, b3);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(rc.empty0 + 8u * stage);
      if (++stage == G::kStages) {
        stage = 0;
        phase ^= 1u;
      }
    }
    // every consumer warp gets here, also when a wait gave up, so that the
    // named barriers below always see all four warps
    consumers_sync();
    if (*rc.abort) break;

    if (P.upt == 1) {
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
      continue;
    }
    float* tile_part = b.partials + P.part_off + (size_t)tile * P.upt * kTile * P.rpad;
    acc_to_partial<R>(tile_part + (size_t)piece * kTile * P.rpad, P.rpad, acc, warp, lane, ntp);
  }
}

// ------------------------------------------------------------------------- column products
template <int R>
__global__ void __launch_bounds__(kThreads) colprod_kernel(const __grid_constant__ ColBatch b) {
  using G = Ring<R>;
  constexpr int NT = R / 8;
  extern __shared__ uint8_t smem_raw[];
  uint32_t base;
  const RingCtl rc = ring_init<R>(smem_raw, &base);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{b.status, b.limit_ns};

  if (warp == kConsumers) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      long long issued = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < b.units && ok; u += gridDim.x) {
        int pi = 0;
        while (pi + 1 < b.n && u >= b.p[pi + 1].unit_begin) ++pi;
        const ColProb& P = b.p[pi];
        const int lu = u - P.unit_begin;
        const int c0 = (lu / P.upt) * kTile;
        const int t_begin = (lu % P.upt) * b.unit_chunks * kTile;
        const int nch = (min(P.T, t_begin + b.unit_chunks * kTile) - t_begin + kTile - 1) / kTile;
        for (int ch = 0; ch < nch; ++ch) {
          const uint32_t empty = rc.empty0 + 8u * stage, full = rc.full0 + 8u * stage;
          if (!mbar_wait(empty, phase ^ 1u, wc, rc.abort)) {
            ok = false;
            break;
          }
          const uint32_t xs = base + (uint32_t)stage * G::kStageBytes;
          const int tb = t_begin + ch * kTile;
          mbar_arrive_expect_tx(full, (uint32_t)P.tx_bytes);
          tma_load_2d(xs, &P.tmX, full, c0, tb);
          int off = 0;
          for (int k = 0; k < P.nblk; ++k) {
            tma_load_2d(xs + kXBytes + (uint32_t)off * (kTile * 2), &P.tmS[k], full, 0, tb);
            off += pad8(P.rs[k]);
          }
          ++issued;
          if (++stage == G::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (*rc.abort) ring_drain<R>(rc, issued);
    }
    return;
  }

  // ------------------------------------------------------------------ consumers
  const int mi = lane >> 3, rr = lane & 7;
  int stage = 0;
  uint32_t phase = 0;
  for (int u = blockIdx.x; u < b.units; u += gridDim.x) {
    int pi = 0;
    while (pi + 1 < b.n && u >= b.p[pi + 1].unit_begin) ++pi;
    const ColProb& P = b.p[pi];
    const int lu = u - P.unit_begin;
    const int tile = lu / P.upt, piece = lu % P.upt;
    const int c0 = tile * kTile;
    const int t_begin = piece * b.unit_chunks * kTile;
    const int nch = (min(P.T, t_begin + b.unit_chunks * kTile) - t_begin + kTile - 1) / kTile;
    const int ntp = P.rpad / 8;
    // rank-side n-tiles: block base (bytes) and row pitch of the tile holding columns 8 n .. 8 n + 7
    uint32_t nbase[NT];
    int npitch[NT];
#pragma unroll
    for (int n = 0; n < NT; ++n) {
      int jj;
      const int bb = find_block(P.rs, P.nblk, n * 8, &jj);
      int off = 0;
      for (int k = 0; k < P.nblk && k < bb; ++k) off += pad8(P.rs[k]);
      npitch[n] = bb >= 0 ? pad8(P.rs[bb]) * 2 : 16;
      nbase[n] = (uint32_t)(off * kTile * 2 + jj * 2);
      if (bb < 0) nbase[n] = 0;
    }

    float acc[NT][4];
#pragma unroll
    for (int n = 0; n < NT; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;

    bool ok = true;
    for (int ch = 0; ch < nch; ++ch) {
      ok = mbar_wait(rc.full0 + 8u * stage, phase, wc, rc.abort);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      const uint32_t xs = base + (uint32_t)stage * G::kStageBytes;
      const uint32_t ss = xs + kXBytes;
#pragma unroll
      for (int ks = 0; ks < kTile / 16; ++ks) {
        // A(m = column c, k = token t) = X[t, c]: the staged tile is k-major, so load transposed
        uint32_t a0, a1, a2, a3;
        ldsm_x4_t(xs + sw128(ks * 16 + (mi >> 1) * 8 + rr, warp * 16 + (mi & 1) * 8), a0, a1, a2, a3);
#pragma unroll
        for (int n = 0; n < NT; n += 2) {
          if (n < ntp) {
            uint32_t b0, b1, b2, b3;
            const int t = ks * 16 + (mi & 1) * 8 + rr;
            const bool hi = (mi >> 1) != 0;  // lanes 16..31 address the second n-tile of the pair
            const uint32_t nb = hi ? nbase[n + 1] : nbase[n];
            const int np = hi ? npitch[n + 1] : npitch[n];
            ldsm_x4_t(ss + nb + (uint32_t)(t * np), b0, b1, b2, b3);
            mma_16816(acc[n], a0, a1, a2, a3, b0, b1);
            mma_16816(acc[n + 1], a0, a1, a2, a3, b2, b3);
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(rc.empty0 + 8u * stage);
      if (++stage == G::kStages) {
        stage = 0;
        phase ^= 1u;
      }
    }
    // every consumer warp gets here, also when a wait gave up, so that the
    // named barriers below always see all four warps
    consumers_sync();
    if (*rc.abort) break;

    if (P.upt == 1) {
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
      continue;
    }
    float* tile_part = b.partials + P.part_off + (size_t)tile * P.upt * kTile * P.rpad;
    acc_to_partial<R>(tile_part + (size_t)piece * kTile * P.rpad, P.rpad, acc, warp, lane, ntp);
  }
}

// Second pass: out = sum of a tile's unit partials, in unit order.  One
// thread per 4 consecutive elements of [tile][64][rpad] of every problem with
// several units (rpad is a multiple of 16, so the 4 share a row); the loads
// of all units are independent and issued together.
template <typename Batch, bool kRow>
__global__ void __launch_bounds__(256) reduce_partials_kernel(const __grid_constant__ Batch b, int total4) {
  const int i4 = blockIdx.x * blockDim.x + threadIdx.x;
  if (i4 >= total4) return;
  const int i = i4 * 4;
  int pi = 0;
  while (pi + 1 < b.n && i >= (int)b.p[pi + 1].red_begin) ++pi;
  const auto& P = b.p[pi];
  const int e = i - P.red_begin;  // element of [tile][64][rpad]
  const int rpad = P.rpad, upt = P.upt;
  const int blk = kTile * rpad;
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
  const int row = tile * kTile + k / rpad, j = k % rpad;
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

// Persistent grid: two CTAs per SM, never more CTAs than units; then the
// reduction pass when any tile has several units.
template <auto Kernel, int R, typename Batch, bool kRow>
cudaError_t launch_units(const Batch& b, int num_sms, cudaStream_t st) {
  constexpr int smem = (int)Ring<R>::kBytes;
  cudaError_t e = set_smem_once<Kernel>(smem);
  if (e != cudaSuccess) return e;
  const int grid = b.units < 2 * num_sms ? b.units : 2 * num_sms;
  Kernel<<<grid, kThreads, smem, st>>>(b);
  note_launch();
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  if (b.red_total > 0) {
    const int total4 = b.red_total / 4;
    reduce_partials_kernel<Batch, kRow><<<(total4 + 255) / 256, 256, 0, st>>>(b, total4);
    note_launch();
    e = cudaGetLastError();
  }
  return e;
}

int grid_for(size_t n, int threads) {
  size_t b = (n + threads - 1) / threads;
  if (b < 1) b = 1;
  if (b > 65535) b = 65535;
  return (int)b;
}

template <int R>
cudaError_t rowprod_r(const RowBatch& b, int num_sms, cudaStream_t st) {
  if (b.w_rc) return launch_units<rowprod_kernel<R, true>, R, RowBatch, true>(b, num_sms, st);
  return launch_units<rowprod_kernel<R, false>, R, RowBatch, true>(b, num_sms, st);
}

}  // namespace

int rank_tile() { return kTile; }

cudaError_t launch_rowprod(const RowBatch& b, int rmax, int num_sms, cudaStream_t st) {
  if (b.n <= 0 || b.units <= 0) return cudaSuccess;
  if (rmax <= 16) return rowprod_r<16>(b, num_sms, st);
  if (rmax <= 32) return rowprod_r<32>(b, num_sms, st);
  if (rmax <= 64) return rowprod_r<64>(b, num_sms, st);
  return rowprod_r<128>(b, num_sms, st);
}

cudaError_t launch_colprod(const ColBatch& b, int rmax, int num_sms, cudaStream_t st) {
  if (b.n <= 0 || b.units <= 0) return cudaSuccess;
  if (rmax <= 16) return launch_units<colprod_kernel<16>, 16, ColBatch, false>(b, num_sms, st);
  if (rmax <= 32) return launch_units<colprod_kernel<32>, 32, ColBatch, false>(b, num_sms, st);
  if (rmax <= 64) return launch_units<colprod_kernel<64>, 64, ColBatch, false>(b, num_sms, st);
  return launch_units<colprod_kernel<128>, 128, ColBatch, false>(b, num_sms, st);
}

cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t st) {
  const size_t n = (size_t)rows * ld_dst;
  pad_cols_kernel<<<grid_for(n, 256), 256, 0, st>>>(src, rows, r, dst, ld_dst);
  note_launch();
  return cudaGetLastError();
}

}  // namespace lora
