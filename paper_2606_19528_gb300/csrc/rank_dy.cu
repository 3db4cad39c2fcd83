// The backward's two rank-r products over dy in one pass (chain rule of the
// LoRA forward y = x W^T + s (x A^T) B^T):
//   sv = s dy B    [T, r]  (bf16; it feeds dx = [dy | sv] [W ; A] and dA = sv^T x)
//   dB = dy^T su   [N, r]  (fp32; su = s x A^T saved by the forward)
// dy is the largest tensor the rank-r work reads; here it is read once.
//
// A CTA (persistent, one per SM) takes work units (token group g, column piece
// q) of one projection.  For each 128-column block of q in turn it streams the
// group's 128-token tiles of dy: one shared-memory stage is a 128-token x
// 128-column tile of dy (two 64-column TMA boxes, 32 KB) with the matching
// boxes of B^T (128 columns) and su^T (128 tokens).  On that stage one thread
// issues two sets of tcgen05.mma (M = 128, N = rpad, K = 16, bf16 -> fp32):
//   sv: A = the dy tile K-major (tokens x columns), B = B^T   -> the tile's sv
//       accumulator, which stays in TMEM for the whole unit;
//   dB: A = the same tile read MN-major (columns x tokens), B = su^T -> the
//       block's dB accumulator, one of two that alternate.
// The epilogue warps drain a dB accumulator as soon as its block has seen every
// token tile of the group, and the sv accumulators when the unit ends.  A
// projection cut into several pieces leaves fp32 sv partials, one cut into
// several token groups fp32 dB partials; a second launch sums them in piece /
// group order, so results never depend on scheduling.  Every wait is bounded.
#include "rank_store.cuh"

namespace lora {

namespace {

constexpr int kTok = 128;                   // tokens per tile: TMEM lanes of an sv accumulator
constexpr int kCols = 128;                  // dy columns per block: TMEM lanes of a dB accumulator
constexpr uint32_t kBox = kTok * 64 * 2;    // one 64-column x 128-token dy box: 16 KB
constexpr uint32_t kDyBytes = 2 * kBox;     // the dy tile of a stage
constexpr int kThreads = 192;               // producer warp, MMA warp, four epilogue warps
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kSmemBudget = 225u * 1024u;  // stages; the control block and alignment take the rest
constexpr int kMaxStages = 8;
constexpr long long kDrainNs = 1000000000ll;

// Rank class R (16, 32, 64, 128 >= rpad): the rank-side box regions hold R
// rows of 128 bytes; TMEM holds kTilesMax sv accumulators of R columns and two
// dB accumulators.
template <int R>
struct DyRing {
  static constexpr uint32_t kSideBox = 128u * R;
  static constexpr uint32_t kStageBytes = kDyBytes + 4 * kSideBox;  // dy, B^T (2 boxes), su^T (2 boxes)
  static constexpr int kStages =
      (int)(kSmemBudget / kStageBytes) < kMaxStages ? (int)(kSmemBudget / kStageBytes) : kMaxStages;
  static constexpr int kTilesMax = (int)(kTmemCols / R) - 2;
  static_assert(kStages >= 2, "two stages at least");
};

struct __align__(8) DyCtl {
  uint64_t full[kMaxStages];
  uint64_t empty[kMaxStages];
  uint64_t dfull[2], dempty[2];  // dB accumulators
  uint64_t sfull, sempty;        // the unit's sv accumulators
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

template <int R>
constexpr size_t dy_smem_bytes() {
  return 1024 + (size_t)DyRing<R>::kStages * DyRing<R>::kStageBytes + sizeof(DyCtl);
}

struct DyUnit {
  int pi, g, q;
  int blk0, blk1;  // column blocks
  int t0, nt;      // first token tile, tiles
};

__device__ __forceinline__ DyUnit dy_unit(const DyBatch& b, int u) {
  DyUnit w;
  w.pi = 0;
  while (w.pi + 1 < b.n && u >= b.p[w.pi + 1].unit_begin) ++w.pi;
  const DyProb& P = b.p[w.pi];
  const int lu = u - P.unit_begin;
  w.g = lu / P.pieces;
  w.q = lu % P.pieces;
  w.blk0 = w.q * P.bpu;
  w.blk1 = min(P.blocks, w.blk0 + P.bpu);
  w.t0 = w.g * P.tt;
  w.nt = min(P.tiles, w.t0 + P.tt) - w.t0;
  return w;
}

// sv elements (t, j .. j + 7), j a multiple of 8 below pad8(r): bf16 of
// scale * v into sv [T, ld_sv] (16-byte store where the layout allows) and
// sv^T [pad8(r), T]; columns r .. pad8(r) - 1 are zeros.
__device__ __forceinline__ void sv_store8(const DyProb& P, int t, int j, const float* v) {
  uint32_t w[4];
#pragma unroll
  for (int e = 0; e < 4; ++e)
    w[e] = pack_bf16x2(j + 2 * e < P.r ? P.scale * v[2 * e] : 0.f, j + 2 * e + 1 < P.r ? P.scale * v[2 * e + 1] : 0.f);
  const __nv_bfloat16* o = reinterpret_cast<const __nv_bfloat16*>(w);
  __nv_bfloat16* d = P.sv + (size_t)t * P.ld_sv + j;
  if ((P.ld_sv & 7) == 0 && j + 8 <= P.ld_sv && aligned16(P.sv)) {
    *reinterpret_cast<uint4*>(d) = make_uint4(w[0], w[1], w[2], w[3]);
  } else {
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (j + e < P.ld_sv) d[e] = o[e];
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) P.svT[(size_t)(j + e) * P.T + t] = o[e];
}

// dB elements (c, j .. j + 15) in fp32 into dB [N, r].
__device__ __forceinline__ void db_store16(const DyProb& P, int c, int j, const float* v) {
  float* d = P.dB + (size_t)c * P.r + j;
  const int n = min(16, P.r - j);
  if (n == 16 && (P.r & 3) == 0 && aligned16(P.dB)) {
#pragma unroll
    for (int e = 0; e < 16; e += 4) reinterpret_cast<float4*>(d)[e / 4] = make_float4(v[e], v[e + 1], v[e + 2], v[e + 3]);
  } else {
#pragma unroll
    for (int e = 0; e < 16; ++e)
      if (e < n) d[e] = v[e];
  }
}

__device__ __forceinline__ void part_store16(float* d, const float* v) {
#pragma unroll
  for (int e = 0; e < 16; e += 4) __stcg(reinterpret_cast<float4*>(d + e), make_float4(v[e], v[e + 1], v[e + 2], v[e + 3]));
}

template <int R>
__global__ void __launch_bounds__(kThreads, 1) rank_dy_kernel(const __grid_constant__ DyBatch b) {
  using G = DyRing<R>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  DyCtl* ctl = reinterpret_cast<DyCtl*>(smem_raw + (base - raw) + (size_t)G::kStages * G::kStageBytes);
  volatile int* abort_flag = &ctl->abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{b.status, b.limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < G::kStages; ++s) {
      mbar_init(smem_u32(&ctl->full[s]), 1);
      mbar_init(smem_u32(&ctl->empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&ctl->dfull[a]), 1);
      mbar_init(smem_u32(&ctl->dempty[a]), 4);  // one arrival per epilogue warp
    }
    mbar_init(smem_u32(&ctl->sfull), 1);
    mbar_init(smem_u32(&ctl->sempty), 4);
    mbar_init(smem_u32(&ctl->drain), 1);
    ctl->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_wait();  // dy, B^T and su^T may come from the previous grid
  const uint32_t tmem_base = ctl->tmem_base;
  long long issued = 0;     // producer: stages issued
  bool issued_any = false;  // MMA issuer: any MMA issued

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < b.units && ok; u += gridDim.x) {
        const DyUnit w = dy_unit(b, u);
        const DyProb& P = b.p[w.pi];
        // full boxes are counted even where they reach past T or N (zero fill)
        const uint32_t tx = kDyBytes + 4u * 64u * 2u * (uint32_t)pad8(P.r);
        for (int blk = w.blk0; blk < w.blk1 && ok; ++blk) {
          const int c0 = blk * kCols;
          for (int j = 0; j < w.nt; ++j) {
            if (!mbar_wait(smem_u32(&ctl->empty[stage]), phase ^ 1u, wc, abort_flag)) {
              ok = false;
              break;
            }
            const uint32_t full = smem_u32(&ctl->full[stage]);
            const uint32_t xs = base + (uint32_t)stage * G::kStageBytes;
            const uint32_t rs = xs + kDyBytes;
            const int tk = (w.t0 + j) * kTok;
            mbar_arrive_expect_tx(full, tx);
            tma_load_2d(xs, &P.tmDy, full, c0, tk);
            tma_load_2d(xs + kBox, &P.tmDy, full, c0 + 64, tk);
            tma_load_2d(rs, &P.tmBt, full, c0, 0);
            tma_load_2d(rs + G::kSideBox, &P.tmBt, full, c0 + 64, 0);
            tma_load_2d(rs + 2 * G::kSideBox, &P.tmSuT, full, tk, 0);
            tma_load_2d(rs + 3 * G::kSideBox, &P.tmSuT, full, tk + 64, 0);
            ++issued;
            if (++stage == G::kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      griddep_launch_dependents();  // every load of this CTA is issued
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int di = 0;  // dB accumulators used so far
      int ui = 0;  // units so far
      bool ok = true;
      // operand descriptors of stage 0 (dy K-major for sv, MN-major for dB; B^T, su^T)
      const uint64_t desc_sv_a = sw128_desc(base, 16, 1024);
      const uint64_t desc_sv_b = sw128_desc(base + kDyBytes, 16, 1024);
      const uint64_t desc_db_a = sw128_desc(base, kBox, 1024);
      const uint64_t desc_db_b = sw128_desc(base + kDyBytes + 2 * G::kSideBox, 16, 1024);
      for (int u = blockIdx.x; u < b.units && ok; u += gridDim.x, ++ui) {
        const DyUnit w = dy_unit(b, u);
        const DyProb& P = b.p[w.pi];
        const uint32_t idesc_sv = idesc_bf16_f32(kTok, P.rpad, 0, 0);
        const uint32_t idesc_db = idesc_bf16_f32(kCols, P.rpad, 1, 0);
        // the previous unit's sv accumulators must be read out first
        if (!mbar_wait(smem_u32(&ctl->sempty), (uint32_t)((ui & 1) ^ 1), wc, abort_flag)) break;
        tc_fence_after();
        for (int blk = w.blk0; blk < w.blk1 && ok; ++blk, ++di) {
          const int buf = di & 1;
          if (!mbar_wait(smem_u32(&ctl->dempty[buf]), (uint32_t)(((di >> 1) & 1) ^ 1), wc, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_db = tmem_base + (uint32_t)((G::kTilesMax + buf) * R);
          for (int j = 0; j < w.nt; ++j) {
            if (!mbar_wait(smem_u32(&ctl->full[stage]), phase, wc, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
            // descriptors of this stage's operands; the steps below only move their start
            // addresses (the address field holds addr >> 4 in its low 14 bits, so adding
            // offset >> 4 within shared memory never carries out of it)
            const uint32_t soff = (uint32_t)stage * (G::kStageBytes >> 4);
            const uint64_t a_sv = desc_sv_a + soff, b_sv = desc_sv_b + soff;
            const uint64_t a_db = desc_db_a + soff, b_db = desc_db_b + soff;
            const uint32_t d_sv = tmem_base + (uint32_t)(j * R);
            const uint32_t acc_sv = blk != w.blk0 ? 1u : 0u, acc_db = j != 0 ? 1u : 0u;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              // sv: 16 columns of dy per step (K-major, box k / 4) against the same columns of B^T
              const uint32_t bx = (uint32_t)(k >> 2), kk = (uint32_t)(k & 3) * 32u;
              umma_bf16(d_sv, a_sv + ((bx * kBox + kk) >> 4), b_sv + ((bx * G::kSideBox + kk) >> 4), idesc_sv,
                        k != 0 ? 1u : acc_sv);
            }
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              // dB: 16 tokens of dy per step (MN-major: the two 64-column boxes kBox apart)
              // against the same tokens of su^T
              const uint32_t bx = (uint32_t)(k >> 2), kk = (uint32_t)(k & 3) * 32u;
              umma_bf16(d_db, a_db + (((uint32_t)k * 2048u) >> 4), b_db + ((bx * G::kSideBox + kk) >> 4), idesc_db,
                        k != 0 ? 1u : acc_db);
            }
            issued_any = true;
            umma_commit(smem_u32(&ctl->empty[stage]));
            if (++stage == G::kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          umma_commit(smem_u32(&ctl->dfull[buf]));
        }
        if (!ok) break;
        umma_commit(smem_u32(&ctl->sfull));
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quadrant: rows q*32 .. q*32+31
    const uint32_t lanes = (uint32_t)(q * 32) << 16;
    int di = 0, ui = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < b.units && ok; u += gridDim.x, ++ui) {
      const DyUnit w = dy_unit(b, u);
      const DyProb& P = b.p[w.pi];
      for (int blk = w.blk0; blk < w.blk1; ++blk, ++di) {
        const int buf = di & 1;
        if (!mbar_wait(smem_u32(&ctl->dfull[buf]), (uint32_t)((di >> 1) & 1), wc, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const int c = blk * kCols + q * 32 + lane;
        const uint32_t taddr = tmem_base + lanes + (uint32_t)((G::kTilesMax + buf) * R);
        float* part = P.groups > 1 ? b.partials + P.db_part + ((size_t)w.g * P.N + c) * P.rpad : nullptr;
#pragma unroll
        for (int j0 = 0; j0 < R; j0 += 16) {
          if (j0 < P.rpad) {  // uniform across the warp
            uint32_t v[16];
            tmem_ld_32x32b_x16(taddr + (uint32_t)j0, v);
            tmem_ld_wait();
            float f[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) f[e] = __uint_as_float(v[e]);
            if (c < P.N) {
              if (part != nullptr)
                part_store16(part + j0, f);
              else if (j0 < P.r)
                db_store16(P, c, j0, f);
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&ctl->dempty[buf]));
      }
      if (!ok) break;
      if (!mbar_wait(smem_u32(&ctl->sfull), (uint32_t)(ui & 1), wc, abort_flag)) break;
      tc_fence_after();
      const int r8 = pad8(P.r);
      for (int j = 0; j < w.nt; ++j) {
        const int t = (w.t0 + j) * kTok + q * 32 + lane;
        const uint32_t taddr = tmem_base + lanes + (uint32_t)(j * R);
        float* part = P.pieces > 1 ? b.partials + P.sv_part + ((size_t)w.q * P.T + t) * P.rpad : nullptr;
#pragma unroll
        for (int j0 = 0; j0 < R; j0 += 16) {
          if (j0 < P.rpad) {
            uint32_t v[16];
            tmem_ld_32x32b_x16(taddr + (uint32_t)j0, v);
            tmem_ld_wait();
            float f[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) f[e] = __uint_as_float(v[e]);
            if (t < P.T) {
              if (part != nullptr) {
                part_store16(part + j0, f);
              } else {
                if (j0 < r8) sv_store8(P, t, j0, f);
                if (j0 + 8 < r8) sv_store8(P, t, j0 + 8, f + 8);
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&ctl->sempty));
    }
  }

  // ---------------------------------------------------------------- teardown
  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // a wait gave up: let this CTA's copies and MMAs complete before its memory is released
    if (warp == 0 && lane == 0) {
      const long long first = issued > G::kStages ? issued - G::kStages : 0;
      for (long long j = first; j < issued; ++j)
        mbar_wait_drain(smem_u32(&ctl->full[j % G::kStages]), (uint32_t)((j / G::kStages) & 1), kDrainNs);
    }
    if (warp == 1 && lane == 0 && issued_any) {
      umma_commit(smem_u32(&ctl->drain));
      mbar_wait_drain(smem_u32(&ctl->drain), 0, kDrainNs);
    }
    tc_fence_before();
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

// Sums the partials of the projections cut into several pieces (sv: in piece
// order, then bf16 of scale * sum into sv and sv^T) or token groups (dB: in
// group order).  A thread takes 8 rank columns of one token's sv (threads in
// turn take consecutive tokens, so the sv^T stores coalesce) or 4 of one dB
// row, and issues the loads of every piece before it sums them.
__global__ void __launch_bounds__(256) dy_reduce_kernel(const __grid_constant__ DyBatch b) {
  griddep_wait();
  const long long total = (long long)b.red_sv + b.red_db;
  for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
       i += (long long)gridDim.x * blockDim.x) {
    long long e = i;
    if (e < b.red_sv) {
      int pi = 0;
      for (; pi < b.n; ++pi) {
        const DyProb& P = b.p[pi];
        if (P.pieces <= 1) continue;
        const long long n = (long long)P.T * (pad8(P.r) / 8);
        if (e < n) break;
        e -= n;
      }
      if (pi >= b.n) continue;  // unreachable with consistent counts
      const DyProb& P = b.p[pi];
      const int j = (int)(e / P.T) * 8, t = (int)(e % P.T);
      const float* src = b.partials + P.sv_part + (size_t)t * P.rpad + j;
      const size_t step = (size_t)P.T * P.rpad;
      float4 lo[kDyMaxCut], hi[kDyMaxCut];
#pragma unroll
      for (int q = 0; q < kDyMaxCut; ++q) {
        if (q < P.pieces) {
          lo[q] = __ldcg(reinterpret_cast<const float4*>(src + q * step));
          hi[q] = __ldcg(reinterpret_cast<const float4*>(src + q * step + 4));
        }
      }
      float v[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int q = 0; q < kDyMaxCut; ++q) {
        if (q < P.pieces) {
          v[0] += lo[q].x, v[1] += lo[q].y, v[2] += lo[q].z, v[3] += lo[q].w;
          v[4] += hi[q].x, v[5] += hi[q].y, v[6] += hi[q].z, v[7] += hi[q].w;
        }
      }
      sv_store8(P, t, j, v);
    } else {
      e -= b.red_sv;
      int pi = 0;
      for (; pi < b.n; ++pi) {
        const DyProb& P = b.p[pi];
        if (P.groups <= 1) continue;
        const long long n = (long long)P.N * ((P.r + 3) / 4);
        if (e < n) break;
        e -= n;
      }
      if (pi >= b.n) continue;  // unreachable with consistent counts
      const DyProb& P = b.p[pi];
      const int jq = (P.r + 3) / 4;
      const int c = (int)(e / jq), j = (int)(e % jq) * 4;
      const float* src = b.partials + P.db_part + (size_t)c * P.rpad + j;
      const size_t step = (size_t)P.N * P.rpad;
      float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int g = 0; g < P.groups; ++g) {
        const float4 a = __ldcg(reinterpret_cast<const float4*>(src + g * step));
        s.x += a.x, s.y += a.y, s.z += a.z, s.w += a.w;
      }
      float* d = P.dB + (size_t)c * P.r + j;
      const float o[4] = {s.x, s.y, s.z, s.w};
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (j + k < P.r) d[k] = o[k];
    }
  }
  griddep_launch_dependents();
}

template <int R>
cudaError_t launch_dy_r(const DyBatch& b, int ctas, cudaStream_t st) {
  constexpr int smem = (int)dy_smem_bytes<R>();
  static std::atomic<unsigned long long> attr_done{0};
  const cudaError_t e = set_smem_once(rank_dy_kernel<R>, smem, attr_done);
  if (e != cudaSuccess) return e;
  const int grid = b.units < ctas ? b.units : ctas;
  return launch_kernel(rank_dy_kernel<R>, dim3(grid), dim3(kThreads), smem, st, 1, b);
}

int rank_class(int rpad) { return rpad <= 16 ? 16 : rpad <= 32 ? 32 : rpad <= 64 ? 64 : 128; }

}  // namespace

int dy_tiles_max(int rpad) { return (int)kTmemCols / rank_class(rpad) - 2; }

cudaError_t launch_dy(const DyBatch& b, int ctas, cudaStream_t st) {
  if (b.n <= 0 || b.units <= 0 || ctas <= 0) return cudaSuccess;
  int rmax = 16;
  for (int i = 0; i < b.n; ++i) rmax = b.p[i].rpad > rmax ? b.p[i].rpad : rmax;
  cudaError_t e;
  switch (rank_class(rmax)) {
    case 16: e = launch_dy_r<16>(b, ctas, st); break;
    case 32: e = launch_dy_r<32>(b, ctas, st); break;
    case 64: e = launch_dy_r<64>(b, ctas, st); break;
    default: e = launch_dy_r<128>(b, ctas, st); break;
  }
  if (e != cudaSuccess || (long long)b.red_sv + b.red_db <= 0) return e;
  const long long total = (long long)b.red_sv + b.red_db;
  const int blocks = (int)std::min<long long>((total + 255) / 256, 8LL * ctas);
  return launch_kernel(dy_reduce_kernel, dim3(blocks), dim3(256), 0, st, 1, b);
}

}  // namespace lora
