// Fused LoRA contraction on the 5th-generation tensor cores (tcgen05, sm_103a).
//
// Forward (Algorithm 1's y_base = W x, extended by the LoRA update):
//     y[T, N]  = [x | su] . [W | B]^T          contraction over K' = K + r
// Backward input gradient (Algorithm 1's dx = W^T dy, extended):
//     dx[T, K] = [dy | sv] . [W ; A]           contraction over N' = N + r
//
// One kernel serves both: the rank-r update is a short tail of extra
// contraction blocks ("adapter slab") appended to the base contraction, so
// base GEMM and update share one fp32 accumulator in tensor memory and the
// output is rounded to bf16 once.  In the forward both operands are K-major
// (x rows and W rows are contiguous along the contraction); in the backward
// the second operand W [N, K] is contracted over its rows, i.e. it is read
// MN-major straight from the frozen weight (no transposed copy of W).
//
// Structure: persistent CTAs (one per SM) take tiles from a tile list
// spanning every problem of a batch (up to kMaxProblems projections, heavier
// first) through a global atomic counter, so that tiles of unequal depth
// balance across SMs; 128 x 256 output tiles, 64-deep contraction blocks.
// Within a problem, consecutive tiles walk M when the weight operand is the
// larger one, so each weight tile is read from DRAM once.
//   warp 0      tile scheduler and TMA producer: 4-stage shared-memory ring,
//               128-byte swizzle
//   warp 1      tcgen05.mma issuer (one thread); owns the TMEM allocation
//   warps 2..5  epilogue: TMEM -> registers -> bf16 -> global
// Two 256-column fp32 accumulators in TMEM (512 columns) let the epilogue of
// one tile overlap the main loop of the next.  Every wait is bounded.
#include "common.cuh"
#include "kernels.h"

namespace lora {

namespace {

constexpr int kBM = 128;
constexpr int kBN = 256;
constexpr int kBK = 64;
constexpr int kStages = 4;
constexpr uint32_t kAStage = kBM * kBK * 2;        // 16 KB
constexpr uint32_t kBStage = kBN * kBK * 2;        // 32 KB
constexpr uint32_t kStageBytes = kAStage + kBStage;
constexpr uint32_t kMnChunk = 64 * kBK * 2;        // one 64-wide MN chunk of B, 8 KB
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr int kTileRing = 4;  // tile ids handed from the producer to the MMA and epilogue warps

struct __align__(8) Ctl {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t tile_full[kTileRing];
  uint64_t tile_empty[kTileRing];
  uint64_t drain;
  int tile_id[kTileRing];
  uint32_t tmem_base;
  int abort;
};

constexpr size_t kSmemBytes = 1024 + (size_t)kStages * kStageBytes + sizeof(Ctl);

__device__ __forceinline__ void decode_tile(const GemmBatch& b, int t, int& p, int& m0, int& n0) {
  p = 0;
  while (p + 1 < b.num_problems && t >= b.prob[p + 1].tile_begin) ++p;
  const GemmProblem& P = b.prob[p];
  const int local = t - P.tile_begin;
  if (P.m_fast) {
    m0 = (local % P.num_m_tiles) * kBM;
    n0 = (local / P.num_m_tiles) * kBN;
  } else {
    m0 = (local / P.num_n_tiles) * kBM;
    n0 = (local % P.num_n_tiles) * kBN;
  }
}

// Consumer side of the tile ring: the id of this role's it-th tile (-1: no more).
__device__ __forceinline__ bool next_tile(Ctl* ctl, int it, const WaitCtl& wc, volatile int* abort, int* t) {
  const int slot = it % kTileRing;
  const uint32_t par = (uint32_t)((it / kTileRing) & 1);
  if (!mbar_wait(smem_u32(&ctl->tile_full[slot]), par, wc, abort)) return false;
  *t = *reinterpret_cast<volatile int*>(&ctl->tile_id[slot]);
  mbar_arrive(smem_u32(&ctl->tile_empty[slot]));
  return true;
}

template <bool kBMn>
__global__ void __launch_bounds__(kThreads, 1) fused_lora_gemm(const __grid_constant__ GemmBatch b) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  Ctl* ctl = reinterpret_cast<Ctl*>(smem_raw + (base - raw) + (size_t)kStages * kStageBytes);
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const WaitCtl wc{b.status, b.limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(smem_u32(&ctl->full[s]), 1);
      mbar_init(smem_u32(&ctl->empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&ctl->tfull[a]), 1);
      mbar_init(smem_u32(&ctl->tempty[a]), 128);
    }
    for (int k = 0; k < kTileRing; ++k) {
      mbar_init(smem_u32(&ctl->tile_full[k]), 1);
      mbar_init(smem_u32(&ctl->tile_empty[k]), 1 + 128);  // MMA thread + epilogue threads
    }
    mbar_init(smem_u32(&ctl->drain), 1);
    ctl->abort = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int p = 0; p < b.num_problems; ++p) {
      tma_prefetch_desc(&b.tmA[p]);
      tma_prefetch_desc(&b.tmA2[p]);
      tma_prefetch_desc(&b.tmB[p]);
      tma_prefetch_desc(&b.tmB2[p]);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = ctl->tmem_base;
  long long issued = 0;     // producer: TMA stage loads issued
  bool issued_any = false;  // MMA issuer: any tcgen05.mma issued

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      for (int it = 0;; ++it) {
        // fetch the next tile and hand its id to the other roles
        const int slot = it % kTileRing;
        if (!mbar_wait(smem_u32(&ctl->tile_empty[slot]), (uint32_t)(((it / kTileRing) & 1) ^ 1), wc, abort_flag))
          break;
        int t = atomicAdd(b.tile_counter, 1);
        if (t >= b.total_tiles) t = -1;
        ctl->tile_id[slot] = t;
        mbar_arrive(smem_u32(&ctl->tile_full[slot]));
        if (t < 0) break;
        int p, m0, n0;
        decode_tile(b, t, p, m0, n0);
        const GemmProblem& P = b.prob[p];
        // backward: 64-wide MN chunks of the weight tile that hold any column < N
        const int chunks = kBMn ? min(4, (P.N - n0 + 63) / 64) : 0;
        const uint32_t tx = kAStage + (kBMn ? (uint32_t)chunks * kMnChunk : kBStage);
        bool ok = true;
        for (int kb = 0; kb < P.kb_total; ++kb) {
          if (!mbar_wait(smem_u32(&ctl->empty[stage]), phase ^ 1u, wc, abort_flag)) {
            ok = false;
            break;
          }
          const uint32_t full = smem_u32(&ctl->full[stage]);
          const uint32_t a_dst = base + stage * kStageBytes;
          const uint32_t b_dst = a_dst + kAStage;
          mbar_arrive_expect_tx(full, tx);
          const bool main = kb < P.kb_main;
          const int kc = main ? kb * kBK : (kb - P.kb_main) * kBK;
          const CUtensorMap* ta = main ? &b.tmA[p] : &b.tmA2[p];
          const CUtensorMap* tb = main ? &b.tmB[p] : &b.tmB2[p];
          tma_load_2d(a_dst, ta, full, kc, m0);
          if (!kBMn) {
            tma_load_2d(b_dst, tb, full, kc, n0);
          } else {
            for (int c = 0; c < chunks; ++c) tma_load_2d(b_dst + c * kMnChunk, tb, full, n0 + 64 * c, kc);
          }
          ++issued;
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN, 0, kBMn ? 1 : 0);
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int it = 0; ok; ++it) {
        int t;
        if (!next_tile(ctl, it, wc, abort_flag, &t) || t < 0) break;
        int p, m0, n0;
        decode_tile(b, t, p, m0, n0);
        const GemmProblem& P = b.prob[p];
        const int acc = it & 1;
        const uint32_t acc_par = (uint32_t)((it >> 1) & 1);
        if (!mbar_wait(smem_u32(&ctl->tempty[acc]), acc_par ^ 1u, wc, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * kBN);
        for (int kb = 0; kb < P.kb_total; ++kb) {
          if (!mbar_wait(smem_u32(&ctl->full[stage]), phase, wc, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = base + stage * kStageBytes;
          const uint32_t b_addr = a_addr + kAStage;
          const int nk = kb < P.kb_main ? kBK / 16 : min(kBK / 16, (P.r - (kb - P.kb_main) * kBK + 15) / 16);
          for (int k = 0; k < nk; ++k) {
            const uint64_t adesc = sw128_desc(a_addr + k * 32, 16, 1024);
            const uint64_t bdesc = kBMn ? sw128_desc(b_addr + k * 2048, kMnChunk, 1024)
                                        : sw128_desc(b_addr + k * 32, 16, 1024);
            umma_bf16(d_tmem, adesc, bdesc, idesc, (kb | k) != 0 ? 1u : 0u);
          }
          issued_any = true;
          umma_commit(smem_u32(&ctl->empty[stage]));
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(smem_u32(&ctl->tfull[acc]));
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;  // TMEM lane quadrant this warp may access
    for (int it = 0;; ++it) {
      int t;
      bool got = next_tile(ctl, it, wc, abort_flag, &t);
      got = __all_sync(0xffffffffu, got);
      if (!got || t < 0) break;
      int p, m0, n0;
      decode_tile(b, t, p, m0, n0);
      const GemmProblem& P = b.prob[p];
      const int acc = it & 1;
      const uint32_t acc_par = (uint32_t)((it >> 1) & 1);
      bool ok = mbar_wait(smem_u32(&ctl->tfull[acc]), acc_par, wc, abort_flag);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      const int row = m0 + q * 32 + lane;
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * kBN);
      __nv_bfloat16* orow = P.out + (size_t)row * P.ldo;
      for (int c = 0; c < kBN; c += 32) {
        if (n0 + c >= P.N) break;  // uniform across the warp
        uint32_t v[32];
        tmem_ld_32x32b_x32(taddr + (uint32_t)c, v);
        tmem_ld_wait();
        if (row < P.M) {
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            const int col = n0 + c + g * 8;
            if (col < P.N) {
              uint4 pk;
              pk.x = pack_bf16x2(__uint_as_float(v[g * 8 + 0]), __uint_as_float(v[g * 8 + 1]));
              pk.y = pack_bf16x2(__uint_as_float(v[g * 8 + 2]), __uint_as_float(v[g * 8 + 3]));
              pk.z = pack_bf16x2(__uint_as_float(v[g * 8 + 4]), __uint_as_float(v[g * 8 + 5]));
              pk.w = pack_bf16x2(__uint_as_float(v[g * 8 + 6]), __uint_as_float(v[g * 8 + 7]));
              *reinterpret_cast<uint4*>(orow + col) = pk;
            }
          }
        }
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&ctl->tempty[acc]));
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // A wait gave up somewhere in the CTA.  Before shared and tensor memory
    // are released, let every copy and MMA this CTA issued complete.
    if (warp == 0 && lane == 0) {
      const long long first = issued > kStages ? issued - kStages : 0;
      for (long long j = first; j < issued; ++j)
        mbar_wait_drain(smem_u32(&ctl->full[j % kStages]), (uint32_t)((j / kStages) & 1), 1000000000ll);
    }
    if (warp == 1 && lane == 0 && issued_any) {
      umma_commit(smem_u32(&ctl->drain));
      mbar_wait_drain(smem_u32(&ctl->drain), 0, 1000000000ll);
    }
    tc_fence_before();
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
}

}  // namespace

size_t fused_gemm_smem_bytes() { return kSmemBytes; }

cudaError_t launch_fused_gemm(const GemmBatch& batch, bool b_mn_major, int num_sms, cudaStream_t stream) {
  static bool attr_done[2] = {false, false};
  const void* fn = b_mn_major ? (const void*)fused_lora_gemm<true> : (const void*)fused_lora_gemm<false>;
  if (!attr_done[b_mn_major]) {
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_done[b_mn_major] = true;
  }
  if (batch.total_tiles <= 0) return cudaSuccess;
  const int grid = batch.total_tiles < num_sms ? batch.total_tiles : num_sms;
  if (b_mn_major)
    fused_lora_gemm<true><<<grid, kThreads, kSmemBytes, stream>>>(batch);
  else
    fused_lora_gemm<false><<<grid, kThreads, kSmemBytes, stream>>>(batch);
  note_launch();
  return cudaGetLastError();
}

int gemm_tile_m() { return kBM; }
int gemm_tile_n() { return kBN; }
int gemm_tile_k() { return kBK; }

}  // namespace lora
