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
// Structure: persistent CTA pairs (thread-block clusters of 2, one CTA per
// SM) take 256 x 512 output tiles from a tile list spanning every problem of
// a batch (up to kMaxProblems projections, heavier first) through a global
// atomic counter, so that tiles of unequal depth balance across SMs.  A tile
// is two 2-CTA tensor-core contractions per 16-deep step (tcgen05
// cta_group::2, M = 256, N = 256 each, one per 256-column segment): each CTA
// of the pair stages its own 128 rows of the activation operand and its own
// 2 x 128 columns of the weight operand, and holds its 128 x 512 half of the
// fp32 accumulator in all 512 columns of its tensor memory.  The wide tile
// halves the shared-memory traffic per FLOP of a 256 x 256 tile, which keeps
// the operand feed ahead of the tensor pipe.  The segments of a tile are
// signalled complete one after the other (the last two blocks issue segment
// 0's MMAs first), and the epilogue drains and releases segment 0 first, so
// the drain of segment 0 overlaps segment 1's last MMAs and the next tile's
// first MMAs overlap the drain of segment 1.  Within a problem, consecutive tiles walk M when the weight
// operand is the larger one, so each weight tile is read from DRAM once.
//   warp 0      tile scheduler (even CTA) and TMA producer (both CTAs):
//               4-stage shared-memory ring of 48 KB, 128-byte swizzle
//   warp 1      TMEM allocation (both CTAs); tcgen05.mma issuer (even CTA)
//   warps 2..9  epilogue: TMEM -> registers -> bf16 -> swizzled shared-memory
//               block (32 rows x 64 columns per warp) -> TMA tensor store
//               (warps 2..5 with 4-bit weights)
// Every wait is bounded.
//
// 4-bit weights (Algorithm 1's on-the-fly dequantization, W = s * W_q + b with
// one (s, b) per output row and 64-wide group along d_in): three decoupled
// rings per CTA.  Warp 0 streams the activation boxes (3 deep); warp 10
// streams this CTA's codes and (s, b) pairs by TMA (a quarter of the bf16
// weight bytes, 2 deep); warps 6..9 dequantize a block with packed bf16
// FMAs straight into the 128-byte-swizzled operand layout the tensor core
// reads, in a ring of 4 bf16 weight tiles, releasing the code slot at once;
// warp 11 relays "tile dequantized" to the MMA issuer (one cluster-scope
// arrive per block and CTA, kept off the dequantizing warps' path); the MMA
// waits for an activation stage and a weight tile.  Each ring has a
// block of slack over its refill latency; the bf16 weight never exists in HBM.
#include "common.cuh"
#include "kernels.h"

namespace lora {

namespace {

constexpr int kBM = 256;                          // tile rows (128 per CTA of a pair)
constexpr int kHalf = 128;
constexpr int kSeg = 256;                         // columns of one MMA / accumulator segment
constexpr int kBN = 2 * kSeg;                     // tile columns
constexpr int kBK = 64;
constexpr uint32_t kAHalf = kHalf * kBK * 2;      // 16 KB: this CTA's activation rows
constexpr uint32_t kBSeg = kHalf * kBK * 2;       // 16 KB: this CTA's weight rows of one segment
constexpr uint32_t kBox = 64 * kBK * 2;           // one 64 x 64 box of the weight operand, 8 KB
constexpr int kEpiWarps = 8;                      // bf16 weights: two per TMEM lane quadrant
constexpr uint32_t kEpiStage = 32 * 128;          // per-warp output block: 32 rows x 64 bf16, 4 KB
constexpr uint32_t kTmemCols = 512;
constexpr int kConvWarps = 4;                     // 4-bit weights: dequantizing warps per CTA

constexpr int kMaxStages = 6;
constexpr uint32_t kStageBytes = kAHalf + 2 * kBSeg;  // bf16 weights: activation + weight boxes
constexpr uint32_t kQCodes = 8192;                    // 4-bit block: 256 weight rows x 64 codes
constexpr uint32_t kQSlot = kQCodes + 4096;           // + (s, b) boxes
constexpr int kQStages = 2;                           // 4-bit: code slots
constexpr int kWStages = 4;                           // 4-bit: dequantized bf16 weight tiles
constexpr uint32_t kWTile = 2 * kBSeg;

// Shared-memory layout and warps of the bf16-weight (kQ false) and
// 4-bit-weight (kQ true) kernels.  bf16: 4 stages of [activation | weight],
// 8 epilogue warps; 4-bit: 3 activation boxes, 4 bf16 weight tiles, 2 code
// slots, 4 epilogue warps (its tiles take longer, so one warp per TMEM lane
// quadrant drains in time) and 4 dequantizing warps.  (4-bit, Llama-shaped
// layer: 4 weight tiles against 3 took T = 256 from 154 to 149 us and T = 2048
// from 731 to 720 us; 2 weight tiles cost 15-30 %; the code ring's depth, 2 to
// 8, changed nothing.)
template <bool kQ>
struct Cfg {
  static constexpr int kStages = kQ ? 3 : 4;  // activation ring
  static constexpr int kEpi = kQ ? 4 : kEpiWarps;
  static constexpr int kParts = kEpi / 4;          // epilogue warps per TMEM lane quadrant
  static constexpr int kPartCols = kSeg / kParts;  // columns of a segment per epilogue warp
  static constexpr uint32_t kRing = kQ ? kStages * kAHalf + kWStages * kWTile + kQStages * kQSlot
                                       : kStages * kStageBytes;
  static constexpr int kThreads = (2 + kEpi + (kQ ? kConvWarps + 2 : 0)) * 32;
  __device__ static uint32_t a_addr(uint32_t base, int s) { return base + (uint32_t)s * (kQ ? kAHalf : kStageBytes); }
  __device__ static uint32_t w_tile(uint32_t base, int w) { return base + kStages * kAHalf + (uint32_t)w * kWTile; }
  __device__ static uint32_t q_slot(uint32_t base, int s) {
    return base + kStages * kAHalf + kWStages * kWTile + (uint32_t)s * kQSlot;
  }
};
constexpr int kTileRing = 4;  // tile ids handed from the scheduler to the other roles
constexpr int kDefer = 2;     // wide tiles: blocks whose segment-0 MMAs precede the first segment-1 MMA
constexpr int kEndDefer = 2;  // wide tiles: last blocks whose segment-0 MMAs precede their segment-1 MMAs
constexpr long long kDrainNs = 1000000000ll;
constexpr long long kAbortDrainNs = 10000000ll;  // 10 ms per armed stage on the abort path

struct __align__(8) Ctl {
  uint64_t full[kMaxStages];       // even CTA: both CTAs' parts of a stage landed
  uint64_t empty[kMaxStages];      // both CTAs: the pair's MMAs finished reading a stage
  uint64_t qfull[kQStages];        // both CTAs, 4-bit: this CTA's codes and (s, b) of a block landed
  uint64_t qempty[kQStages];       // both CTAs, 4-bit: this CTA's dequantizers read a code slot
  uint64_t wfull[kWStages];        // even CTA, 4-bit: both CTAs' weight tile dequantized (or loaded)
  uint64_t convd[kWStages];        // both CTAs, 4-bit: this CTA's dequantizing warps finished a weight tile
  uint64_t wempty[kWStages];       // both CTAs, 4-bit: the pair's MMAs finished reading a weight tile
  uint64_t tfull[2];               // both CTAs: accumulator (buffer) complete
  uint64_t tempty[2];              // even CTA: both CTAs' epilogues drained a segment (buffer)
  uint64_t tile_full[kTileRing];   // both CTAs: tile id written
  uint64_t tile_empty[kTileRing];  // even CTA: every consumer of both CTAs read the slot
  uint64_t drain;                  // both CTAs: every MMA of the pair completed
  uint64_t xchg;                   // kCS: the other pair's half of the accumulator arrived
  int tile_id[kTileRing];
  uint32_t tmem_base;
  int abort;
  int fills;   // ring stages this CTA's producer armed (expect_tx on the even CTA's barriers)
  int qfills;  // 4-bit: code slots this CTA's code producer armed
};

template <bool kQ>
constexpr size_t smem_bytes() {
  return 1024 + (size_t)Cfg<kQ>::kRing + (size_t)Cfg<kQ>::kEpi * kEpiStage + sizeof(Ctl);
}

// Problem p, first row m0 and first column n0 of tile t, its split ks and
// that split's contraction blocks [kb0, kb1).  cs_half >= 0 (cluster split):
// the tile is unsplit in the list and the pair takes half cs_half of its
// contraction blocks (the first half rounded up).
template <int kTileN = kBN>
__device__ __forceinline__ void decode_tile(const GemmBatch& b, int t, int& p, int& m0, int& n0, int& ks, int& kb0,
                                            int& kb1, int cs_half = -1) {
  p = 0;
  while (p + 1 < b.num_problems && t >= b.prob[p + 1].tile_begin) ++p;
  const GemmProblem& Q = b.prob[p];
  int local = t - Q.tile_begin;
  const int per = Q.num_m_tiles * Q.num_n_tiles;
  ks = local / per;
  local -= ks * per;
  kb0 = ks * Q.kb_split;
  kb1 = min(Q.kb_total, kb0 + Q.kb_split);
  if (cs_half >= 0) {
    const int L = (Q.kb_total + 1) / 2;
    kb0 = cs_half * L;
    kb1 = min(Q.kb_total, kb0 + L);
  }
  if (Q.m_fast) {
    m0 = (local % Q.num_m_tiles) * kBM;
    n0 = (local / Q.num_m_tiles) * kTileN;
  } else {
    m0 = (local / Q.num_n_tiles) * kBM;
    n0 = (local % Q.num_n_tiles) * kTileN;
  }
}

// Two 4-bit codes -> bf16x2 (s * q + b): the codes sit at bits 0..3 and
// 16..19 of `w`; OR-ing in the exponent of 128 gives exactly 128 + q per half,
// the first FMA takes 128 off (exact), the second rounds s * q + b once.
__device__ __forceinline__ uint32_t dq_pair(uint32_t w, uint32_t s2, uint32_t b2) {
  const uint32_t v = (w & 0x000F000Fu) | 0x43004300u;
  uint32_t q, r;
  asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(q) : "r"(v), "r"(0x3F803F80u), "r"(0xC300C300u));
  asm("fma.rn.bf16x2 %0, %1, %2, %3;" : "=r"(r) : "r"(q), "r"(s2), "r"(b2));
  return r;
}

// Dequantizes this CTA's weight operand of one contraction block from the
// staged codes and (s, b) pairs into the 128-byte-swizzled bf16 boxes the MMA
// reads.  Row rho of box (h, j) is weight column / row col0 = n0 + 256 h +
// 128 c + 64 j of the tile: the forward's rows are W rows col0 + rho at
// k-group kb; the backward's are W rows 64 kb + rho at k-group col0 / 64.
// Staged boxes: forward, codes (h, j) 64 rows x 32 B at 2 KB (2 h + j), (s, b)
// h 128 rows x 4 groups at 2 KB h; backward, codes h 64 rows x 64 B at 4 KB h,
// (s, b) h 64 rows x 4 groups at 1 KB h.  A thread takes half rows (32 codes,
// 16 bytes) ordered so that a warp reads 512 contiguous bytes of codes.
template <bool kBMn>
__device__ __forceinline__ void dequant_stage(uint32_t slot, uint32_t wdst, int ct, int c, int n0, int kb,
                                              int ncols) {
  constexpr int kThr = kConvWarps * 32;
  const uint32_t codes = slot;
  const uint32_t params = slot + kQCodes;
#pragma unroll
  for (int rep = 0; rep < 512 / kThr; ++rep) {
    const int hu = ct + rep * kThr;  // half row
    const int half = hu & 1, h = hu >> 8;
    const int j = kBMn ? (hu >> 1) & 1 : (hu >> 7) & 1;
    const int rho = kBMn ? (hu >> 2) & 63 : (hu >> 1) & 63;
    const int colh = n0 + h * kSeg + c * kHalf;
    if (colh + j * 64 >= ncols) continue;  // box not loaded: its MMA columns are never stored
    uint32_t csrc, psrc;
    if (kBMn) {
      const int g = (colh >> 6) + j, gb = (colh >> 6) & ~3;
      csrc = codes + (uint32_t)(h * 4096 + rho * 64 + j * 32 + half * 16);
      psrc = params + (uint32_t)(h * 1024 + rho * 16 + (g - gb) * 4);
    } else {
      csrc = codes + (uint32_t)((h * 2 + j) * 2048 + rho * 32 + half * 16);
      psrc = params + (uint32_t)(h * 2048 + (j * 64 + rho) * 16 + (kb & 3) * 4);
    }
    uint32_t w[4], sb;
    asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(w[0]), "=r"(w[1]), "=r"(w[2]), "=r"(w[3]) : "r"(csrc) : "memory");
    asm volatile("ld.shared.b32 %0, [%1];" : "=r"(sb) : "r"(psrc) : "memory");
    const uint32_t s2 = (sb & 0xFFFFu) * 0x10001u, b2 = (sb >> 16) * 0x10001u;
    const uint32_t row = wdst + (uint32_t)(h * kBSeg + j * kBox + rho * 128);
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      const uint32_t o0 = dq_pair(w[m], s2, b2), o1 = dq_pair(w[m] >> 4, s2, b2);
      const uint32_t o2 = dq_pair(w[m] >> 8, s2, b2), o3 = dq_pair(w[m] >> 12, s2, b2);
      const uint32_t dst = row + (uint32_t)((((half * 4 + m) ^ (rho & 7)) & 7) << 4);
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(o0), "r"(o1), "r"(o2), "r"(o3)
                   : "memory");
    }
  }
}

template <bool kBMn, bool kQ, bool kF32 = false, bool kCS = false>
__global__ void __launch_bounds__(Cfg<kQ>::kThreads, 1) fused_lora_gemm(const __grid_constant__ GemmBatch b) {
  // fp32 output: 256 x 256 tiles whose accumulator alternates between two TMEM
  // buffers, so one tile's epilogue overlaps the next tile's contraction (the
  // appending and log-sum-exp epilogues are long); a 6-deep ring of 32 KB stages.
  // kCS (cluster split, bf16 output): clusters of two CTA pairs, one 256 x 256
  // tile per cluster; pair j contracts half j of the tile's blocks, then the
  // halves are summed through distributed shared memory (each pair finishes
  // and stores its own 128 columns): no fp32 partials in global memory, no
  // reduce launch.  For launches with too few tiles to fill the GPU.
  constexpr bool kNarrow = kF32 || kCS;
  static_assert(!kNarrow || !kQ, "256 x 256 tiles: bf16 weights only");
  static_assert(!kF32 || (!kBMn && !kCS), "fp32 output is the plain forward form");
  constexpr int kSegs = kNarrow ? 1 : 2;  // 256-column segments per tile
  constexpr int kTileN = kSegs * kSeg;
  constexpr int kStages = kNarrow ? 6 : Cfg<kQ>::kStages;
  constexpr uint32_t kStageB = kNarrow ? kAHalf + kBSeg : kStageBytes;
  static_assert(kStages <= kMaxStages && (!kNarrow || kStages * kStageB <= Cfg<kQ>::kRing), "ring");
  auto a_addr_of = [&](uint32_t bs, int st) {
    return kQ ? Cfg<kQ>::a_addr(bs, st) : bs + (uint32_t)st * kStageB;
  };
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t epi_base = base + Cfg<kQ>::kRing;  // 1024-aligned output staging blocks
  constexpr int kEpi = Cfg<kQ>::kEpi;
  Ctl* ctl = reinterpret_cast<Ctl*>(smem_raw + (base - raw) + (size_t)Cfg<kQ>::kRing + (size_t)kEpi * kEpiStage);
  volatile int* abort_flag = &ctl->abort;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t crank = cluster_ctarank();
  const int c = (int)(crank & 1u);  // position within the pair (0: issues the MMAs)
  const uint32_t pb = crank & ~1u;  // cluster rank of the pair's even CTA (0 but for kCS)
  const int cs_half = kCS ? (int)((crank >> 1) & 1u) : -1;  // kCS: which half of the contraction
  const int cs_tile = kCS ? (int)(blockIdx.x >> 2) : 0;     // kCS: the cluster's one tile
  const WaitCtl wc{b.status, b.limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      // producer (expect_tx), plus every dequantizing warp of both CTAs
      mbar_init(smem_u32(&ctl->full[s]), 1);
      mbar_init(smem_u32(&ctl->empty[s]), 1);
    }
    for (int q = 0; q < kQStages; ++q) {
      mbar_init(smem_u32(&ctl->qfull[q]), 1);
      mbar_init(smem_u32(&ctl->qempty[q]), kConvWarps);
    }
    for (int w = 0; w < kWStages; ++w) {
      mbar_init(smem_u32(&ctl->wfull[w]), 2);  // the relay of each CTA
      mbar_init(smem_u32(&ctl->convd[w]), kConvWarps);
      mbar_init(smem_u32(&ctl->wempty[w]), 1);
    }
    mbar_init(smem_u32(&ctl->tfull[0]), 1);
    mbar_init(smem_u32(&ctl->tfull[1]), 1);
    for (int h = 0; h < 2; ++h) mbar_init(smem_u32(&ctl->tempty[h]), 2 * kEpi);
    for (int k = 0; k < kTileRing; ++k) {
      mbar_init(smem_u32(&ctl->tile_full[k]), 1);
      // MMA thread, epilogue (and dequantizing, code producer, relay) warps of both CTAs, producer of the odd CTA
      mbar_init(smem_u32(&ctl->tile_empty[k]), 2 + 2 * kEpi + (kQ ? 2 * kConvWarps + 4 : 0));
    }
    mbar_init(smem_u32(&ctl->drain), 1);
    mbar_init(smem_u32(&ctl->xchg), 1);
    ctl->abort = 0;
    ctl->fills = 0;
    ctl->qfills = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    for (int q = 0; q < b.num_problems; ++q) {
      tma_prefetch_desc(&b.tmA[q]);
      tma_prefetch_desc(&b.tmA2[q]);
      if (kQ) {
        tma_prefetch_desc(&b.tmQ[q]);
        tma_prefetch_desc(&b.tmP[q]);
      } else {
        tma_prefetch_desc(&b.tmB[q]);
      }
      tma_prefetch_desc(&b.tmB2[q]);
      tma_prefetch_desc(&b.tmOut[q]);
    }
  }
  if (warp == 1) {
    tmem_alloc_pair(smem_u32(&ctl->tmem_base), kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  cluster_sync_all();  // both CTAs' barriers exist before any cross-CTA arrival
  // the previous grid's outputs (su, sv) are ready; with early inputs only the producer waits, before its
  // first adapter-slab load (the tile counter was cleared before the call's first kernel)
  if (!b.early_inputs) griddep_wait();
  const uint32_t tmem_base = ctl->tmem_base;
  const uint32_t tile_empty_root = mapa_shared(smem_u32(&ctl->tile_empty[0]), pb);

  if (warp == 0) {
    // ------------------------------------------------------------ scheduler + producer
    if (lane == 0) {
      const uint32_t full_pl = mapa_shared(smem_u32(&ctl->full[0]), pb);
      int stage = 0;
      uint32_t phase = 0;
      int fills = 0;
      bool waited = !b.early_inputs;  // this thread has waited for the previous grid
      for (int it = 0;; ++it) {
        const int slot = it % kTileRing;
        const uint32_t par = (uint32_t)((it / kTileRing) & 1);
        int t;
        if (kCS) {
          t = it == 0 ? cs_tile : -1;  // one tile, no scheduler
        } else if (c == 0) {
          if (!mbar_wait_cluster(smem_u32(&ctl->tile_empty[slot]), par ^ 1u, wc, abort_flag)) break;
          t = atomicAdd(b.tile_counter, 1);
          if (t >= b.total_tiles) t = -1;
          ctl->tile_id[slot] = t;
          st_cluster_u32(mapa_shared(smem_u32(&ctl->tile_id[slot]), pb + 1), (uint32_t)t);
          mbar_arrive(smem_u32(&ctl->tile_full[slot]));
          mbar_arrive_cluster(mapa_shared(smem_u32(&ctl->tile_full[slot]), pb + 1));
        } else {
          if (!mbar_wait_cluster(smem_u32(&ctl->tile_full[slot]), par, wc, abort_flag)) break;
          t = *reinterpret_cast<volatile int*>(&ctl->tile_id[slot]);
          mbar_arrive_cluster(tile_empty_root + (uint32_t)slot * 8u);
        }
        if (t < 0) {
          griddep_launch_dependents();  // no tile left for this pair
          break;
        }
        int p, m0, n0, ks, kb0, kb1;
        decode_tile<kTileN>(b, t, p, m0, n0, ks, kb0, kb1, cs_half);
        const GemmProblem& Q = b.prob[p];
        const int my_m = m0 + c * kHalf;
        const bool a_mine = my_m < Q.M;
        // weight box (segment h, pair position cc, j): columns n0 + 256 h + 128 cc + 64 j
        auto box_ok = [&](int h, int cc, int j) { return n0 + h * kSeg + cc * kHalf + j * 64 < Q.N; };
        uint32_t boxes = 0;
        for (int h = 0; h < kSegs; ++h)
          for (int cc = 0; cc < 2; ++cc)
            for (int j = 0; j < 2; ++j) boxes += box_ok(h, cc, j) ? 1u : 0u;
        // bytes landing in this pair per stage (signalled on the even CTA)
        const uint32_t tx_a = (m0 < Q.M ? kAHalf : 0u) + (m0 + kHalf < Q.M ? kAHalf : 0u);
        const uint32_t tx_pair = tx_a + kBox * boxes;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait_cluster(smem_u32(&ctl->empty[stage]), phase ^ 1u, wc, abort_flag)) {
            ok = false;
            break;
          }
          const bool main = kb < Q.kb_main;
          // with 4-bit weights the dequantizing warps fill the weight tiles
          const bool w_tma = !kQ;
          if (c == 0) mbar_arrive_expect_tx(smem_u32(&ctl->full[stage]), w_tma ? tx_pair : tx_a);
          ++fills;
          const uint32_t bar = full_pl + (uint32_t)stage * 8u;
          const uint32_t a_dst = a_addr_of(base, stage);
          const uint32_t b_dst = a_dst + kAHalf;
          const int kc = main ? kb * kBK : (kb - Q.kb_main) * kBK;
          if (!main && !waited) {
            griddep_wait();  // su or sv comes from the previous grid
            waited = true;
          }
          const CUtensorMap* ta = main ? &b.tmA[p] : &b.tmA2[p];
          const CUtensorMap* tb = main ? &b.tmB[p] : &b.tmB2[p];
          if (a_mine) tma_load_2d_pair(a_dst, ta, bar, kc, my_m);
          if (w_tma) {
#pragma unroll
            for (int h = 0; h < kSegs; ++h) {
#pragma unroll
              for (int j = 0; j < 2; ++j) {
                if (!box_ok(h, c, j)) continue;
                const int col = n0 + h * kSeg + c * kHalf + j * 64;
                tma_load_2d_pair(b_dst + h * kBSeg + j * kBox, tb, bar, kBMn ? col : kc, kBMn ? kc : col);
              }
            }
          }
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      ctl->fills = fills;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (even CTA)
    if (c == 0 && lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, kSeg, 0, kBMn ? 1 : 0);
      const uint16_t pair_mask = (uint16_t)(0x3u << pb);
      int stage = 0;
      uint32_t phase = 0;
      uint32_t wseq = 0;  // 4-bit: contraction blocks so far (weight tile wseq % 2)
      bool ok = true;
      for (int it = 0; ok; ++it) {
        const int slot = it % kTileRing;
        int t;
        if (kCS) {
          t = it == 0 ? cs_tile : -1;
        } else {
          if (!mbar_wait_cluster(smem_u32(&ctl->tile_full[slot]), (uint32_t)((it / kTileRing) & 1), wc, abort_flag))
            break;
          t = *reinterpret_cast<volatile int*>(&ctl->tile_id[slot]);
          mbar_arrive_cluster(tile_empty_root + (uint32_t)slot * 8u);
        }
        if (t < 0) {
          griddep_launch_dependents();  // no tile left for this pair
          break;
        }
        int p, m0, n0, ks, kb0, kb1;
        decode_tile<kTileN>(b, t, p, m0, n0, ks, kb0, kb1, cs_half);
        const GemmProblem& Q = b.prob[p];
        const int nseg = kNarrow ? 1 : (Q.N - n0 > kSeg ? 2 : 1);  // segments holding any column < N
        // accumulator buffer of this tile; a segment (buffer) is free once both epilogues drained
        // it for its previous tile (the previous tile, or with two buffers the one before)
        const int buf = kNarrow ? (it & 1) : 0;
        const uint32_t drained_par = kNarrow ? (uint32_t)(((it >> 1) & 1) ^ 1) : (uint32_t)((it & 1) ^ 1);
        int kb = kb0;
        if (!kQ && kSegs == 2) {
          // Start of a wide tile: segment 0's MMAs of the first kDefer blocks go first, and only then
          // does the issuer need segment 1's accumulator (the epilogue drains segment 0 first).  Each
          // segment still accumulates its blocks in order, so the sums are unchanged.
          const int nd = min(kDefer, kb1 - kb0);
          int dst[kDefer];
          for (int i = 0; i < nd && ok; ++i, ++kb) {
            if (!mbar_wait(smem_u32(&ctl->full[stage]), phase, wc, abort_flag) ||
                (i == 0 && !mbar_wait_cluster(smem_u32(&ctl->tempty[buf]), drained_par, wc, abort_flag))) {
              ok = false;
              break;
            }
            tc_fence_after();
            dst[i] = stage;
            const uint32_t a_addr = a_addr_of(base, stage);
            const int nk = kb < Q.kb_main ? kBK / 16 : min(kBK / 16, (Q.r - (kb - Q.kb_main) * kBK + 15) / 16);
            const uint64_t ad = sw128_desc(a_addr, 16, 1024);
            const uint64_t bd = kBMn ? sw128_desc(a_addr + kAHalf, kBox, 1024) : sw128_desc(a_addr + kAHalf, 16, 1024);
            for (int k = 0; k < nk; ++k)
              umma_bf16_pair(tmem_base + (uint32_t)(buf * kSeg), ad + (uint64_t)(2 * k),
                             bd + (uint64_t)((kBMn ? 128 : 2) * k), idesc, (kb != kb0 || k != 0) ? 1u : 0u);
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (ok && !mbar_wait_cluster(smem_u32(&ctl->tempty[buf + 1]), drained_par, wc, abort_flag)) ok = false;
          if (!ok) break;
          tc_fence_after();
          for (int i = 0; i < nd; ++i) {
            const int kbi = kb0 + i;
            const uint32_t a_addr = a_addr_of(base, dst[i]);
            const int nk = kbi < Q.kb_main ? kBK / 16 : min(kBK / 16, (Q.r - (kbi - Q.kb_main) * kBK + 15) / 16);
            if (nseg > 1) {
              const uint64_t ad = sw128_desc(a_addr, 16, 1024);
              const uint64_t bd = kBMn ? sw128_desc(a_addr + kAHalf + kBSeg, kBox, 1024)
                                       : sw128_desc(a_addr + kAHalf + kBSeg, 16, 1024);
              for (int k = 0; k < nk; ++k)
                umma_bf16_pair(tmem_base + (uint32_t)((buf + 1) * kSeg), ad + (uint64_t)(2 * k),
                               bd + (uint64_t)((kBMn ? 128 : 2) * k), idesc, (kbi != kb0 || k != 0) ? 1u : 0u);
            }
            umma_commit_pair_mc(smem_u32(&ctl->empty[dst[i]]), pair_mask);
          }
        }
        // wide bf16 tiles with both segments: the last kEndDefer blocks are issued below
        const int kb_end = (!kQ && kSegs == 2 && nseg == 2 && kb1 - kb >= kEndDefer) ? kb1 - kEndDefer : kb1;
        for (; kb < kb_end; ++kb) {
          if (!mbar_wait(smem_u32(&ctl->full[stage]), phase, wc, abort_flag)) {
            ok = false;
            break;
          }
          const int wt = (int)(wseq % kWStages);
          if (kQ && !mbar_wait_cluster(smem_u32(&ctl->wfull[wt]), (wseq / kWStages) & 1u, wc, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = a_addr_of(base, stage);
          const uint32_t b_addr = kQ ? Cfg<kQ>::w_tile(base, wt) : a_addr + kAHalf;
          const int nk = kb < Q.kb_main ? kBK / 16 : min(kBK / 16, (Q.r - (kb - Q.kb_main) * kBK + 15) / 16);
          if (kb != kb0 && nk == kBK / 16 && nseg == kSegs) {
            // Steady state (every segment, full depth, accumulating).  The one issuing thread paces
            // the main loop, so its instructions per MMA are kept to a minimum: each operand's
            // descriptor is built once per block and advanced by the 16-deep step in its start-address
            // field (address >> 4; 32 bytes of a K-major row, 2048 bytes = 16 rows of an MN-major
            // operand; shared addresses stay below the field's 2^18-byte range).  The same MMAs as the
            // general form below; this form took the Llama-shaped layer's two contractions from 271 /
            // 251 us to 242 / 232 us per step.
            const uint64_t ad = sw128_desc(a_addr, 16, 1024);
#pragma unroll
            for (int h = 0; h < kSegs; ++h) {
              const uint64_t bd = kBMn ? sw128_desc(b_addr + (uint32_t)h * kBSeg, kBox, 1024)
                                       : sw128_desc(b_addr + (uint32_t)h * kBSeg, 16, 1024);
#pragma unroll
              for (int k = 0; k < kBK / 16; ++k)
                umma_bf16_pair(tmem_base + (uint32_t)((buf + h) * kSeg), ad + (uint64_t)(2 * k),
                               bd + (uint64_t)((kBMn ? 128 : 2) * k), idesc, 1u);
            }
          } else
          for (int h = 0; h < kSegs; ++h) {
            if (kb == kb0) {
              if (!mbar_wait_cluster(smem_u32(&ctl->tempty[buf + h]), drained_par, wc, abort_flag)) {
                ok = false;
                break;
              }
              tc_fence_after();
            }
            if (h >= nseg) continue;
            const uint32_t d_tmem = tmem_base + (uint32_t)((buf + h) * kSeg);
            const uint32_t bseg = b_addr + (uint32_t)h * kBSeg;
            for (int k = 0; k < nk; ++k) {
              const uint64_t adesc = sw128_desc(a_addr + k * 32, 16, 1024);
              const uint64_t bdesc = kBMn ? sw128_desc(bseg + k * 2048, kBox, 1024) : sw128_desc(bseg + k * 32, 16, 1024);
              umma_bf16_pair(d_tmem, adesc, bdesc, idesc, (kb != kb0 || k != 0) ? 1u : 0u);
            }
          }
          if (!ok) break;
          umma_commit_pair_mc(smem_u32(&ctl->empty[stage]), pair_mask);
          if (kQ) umma_commit_pair_mc(smem_u32(&ctl->wempty[wt]), pair_mask);
          ++wseq;
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        if (kSegs == 2) {
          // End of a wide tile: segment 0's MMAs of the last blocks go first and segment 0 is signalled
          // complete before segment 1, so its drain overlaps segment 1's last MMAs.  Each segment still
          // accumulates its blocks in order.
          int dst2[kEndDefer];
          const int ne = kQ ? 0 : kb1 - kb;
          for (int i = 0; i < ne && ok; ++i, ++kb) {
            if (!mbar_wait(smem_u32(&ctl->full[stage]), phase, wc, abort_flag)) {
              ok = false;
              break;
            }
            tc_fence_after();
            dst2[i] = stage;
            const uint32_t a_addr = a_addr_of(base, stage);
            const int nk = kb < Q.kb_main ? kBK / 16 : min(kBK / 16, (Q.r - (kb - Q.kb_main) * kBK + 15) / 16);
            const uint64_t ad = sw128_desc(a_addr, 16, 1024);
            const uint64_t bd = kBMn ? sw128_desc(a_addr + kAHalf, kBox, 1024) : sw128_desc(a_addr + kAHalf, 16, 1024);
            for (int k = 0; k < nk; ++k)
              umma_bf16_pair(tmem_base, ad + (uint64_t)(2 * k), bd + (uint64_t)((kBMn ? 128 : 2) * k), idesc, 1u);
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          umma_commit_pair_mc(smem_u32(&ctl->tfull[0]), pair_mask);
          for (int i = 0; i < ne; ++i) {
            const int kbi = kb1 - ne + i;
            const uint32_t a_addr = a_addr_of(base, dst2[i]);
            const int nk = kbi < Q.kb_main ? kBK / 16 : min(kBK / 16, (Q.r - (kbi - Q.kb_main) * kBK + 15) / 16);
            const uint64_t ad = sw128_desc(a_addr, 16, 1024);
            const uint64_t bd = kBMn ? sw128_desc(a_addr + kAHalf + kBSeg, kBox, 1024)
                                     : sw128_desc(a_addr + kAHalf + kBSeg, 16, 1024);
            for (int k = 0; k < nk; ++k)
              umma_bf16_pair(tmem_base + (uint32_t)kSeg, ad + (uint64_t)(2 * k), bd + (uint64_t)((kBMn ? 128 : 2) * k),
                             idesc, 1u);
            umma_commit_pair_mc(smem_u32(&ctl->empty[dst2[i]]), pair_mask);
          }
          umma_commit_pair_mc(smem_u32(&ctl->tfull[1]), pair_mask);
        } else {
          umma_commit_pair_mc(smem_u32(&ctl->tfull[buf]), pair_mask);
        }
      }
      // completes in both CTAs of the pair once every MMA issued above has finished
      umma_commit_pair_mc(smem_u32(&ctl->drain), pair_mask);
    }
  } else if (kCS && warp < 2 + kEpi) {
    // ------------------------------------------------------------ epilogue, cluster split: wait for the
    // pair's accumulator; the exchange of the halves follows below, after every role
    bool ok = mbar_wait_cluster(smem_u32(&ctl->tfull[0]), 0u, wc, abort_flag);
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();
  } else if (warp < 2 + kEpi) {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int q = warp & 3;                 // TMEM lane quadrant this warp may access
    const int part = (warp - 2) >> 2;       // which kPartCols columns of each segment
    const uint32_t tempty_pl = mapa_shared(smem_u32(&ctl->tempty[0]), pb);
    for (int it = 0;; ++it) {
      const int slot = it % kTileRing;
      bool got = mbar_wait_cluster(smem_u32(&ctl->tile_full[slot]), (uint32_t)((it / kTileRing) & 1), wc, abort_flag);
      got = __all_sync(0xffffffffu, got);
      if (!got) break;
      const int t = *reinterpret_cast<volatile int*>(&ctl->tile_id[slot]);
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tile_empty_root + (uint32_t)slot * 8u);
      if (t < 0) break;
      int p, m0, n0, ks, kb0, kb1;
      decode_tile<kTileN>(b, t, p, m0, n0, ks, kb0, kb1);
      const GemmProblem& Q = b.prob[p];
      const int buf = kNarrow ? (it & 1) : 0;  // accumulator buffer of this tile
      const uint32_t tpar = kNarrow ? (uint32_t)((it >> 1) & 1) : (uint32_t)(it & 1);
      // wide tiles signal each segment's accumulator complete on its own (tfull[h])
      bool ok = kSegs == 2 || mbar_wait_cluster(smem_u32(&ctl->tfull[buf]), tpar, wc, abort_flag);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      const int row0 = m0 + c * kHalf + q * 32;  // first of this warp's 32 rows
      const uint32_t stg = epi_base + (uint32_t)(warp - 2) * kEpiStage;
      for (int h = 0; h < kSegs; ++h) {
        if (kSegs == 2) {
          bool okh = mbar_wait_cluster(smem_u32(&ctl->tfull[h]), tpar, wc, abort_flag);
          okh = __all_sync(0xffffffffu, okh);
          if (!okh) {
            ok = false;
            break;
          }
          tc_fence_after();
        }
        // a staged block is 32 rows x 128 bytes: 64 bf16 columns, or 32 fp32 columns
        // (fp32 output, or the partial of one split of the contraction)
        const bool f32 = kF32 || Q.splits > 1;
        const int block_cols = f32 ? 32 : 64;
        const int row_st = (Q.splits > 1 ? ks * Q.m_pad : 0) + row0;  // stored row of this warp's first row
        // log-sum-exp partial of this thread's row over the warp's column group
        const bool lse_on = kF32 && Q.lse != nullptr && Q.splits == 1;  // split partials: the reduce does it
        const bool app = kF32 && Q.cand != nullptr;  // append mode (never split)
        const float tau = app && row0 + lane < Q.M ? Q.tau[Q.row_off + row0 + lane] : INFINITY;
        float lm = -INFINITY, ls = 0.f;
        if (app && row0 < Q.M && n0 + h * kSeg + part * Cfg<kQ>::kPartCols < Q.N) {  // uniform across the warp
          // append mode: a first pass over the warp's columns records hits as bit masks (this
          // thread's row; with the transposed side also lane l's column of each 32-column
          // block, over the warp's 32 rows), one atomic per list reserves the slots, a second
          // pass writes the hits
          constexpr int kBlocks = Cfg<kQ>::kPartCols / 32;
          const bool tr = Q.sym && n0 >= kSymRows;  // off the diagonal block
          const int i_abs = Q.row_off + row0 + lane;
          // the transposed side reads the block column-wise from the warp's staging buffer
          // (free in append mode): row `lane` stored as 8 16-byte chunks, chunk u at u ^ (lane mod 8)
          auto stage_block = [&](const uint32_t(&v)[32]) {
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              const uint32_t a = stg + (uint32_t)lane * 128u + (uint32_t)(((u ^ (lane & 7)) & 7) << 4);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(v[4 * u]), "r"(v[4 * u + 1]),
                           "r"(v[4 * u + 2]), "r"(v[4 * u + 3])
                           : "memory");
            }
            __syncwarp();
          };
          auto col_value = [&](int r) {  // row r, column `lane` of the staged block
            const uint32_t a = stg + (uint32_t)r * 128u + (uint32_t)((((lane >> 2) ^ (r & 7)) & 7) << 4) +
                               (uint32_t)(lane & 3) * 4u;
            float x;
            asm volatile("ld.shared.f32 %0, [%1];" : "=f"(x) : "r"(a) : "memory");
            return x;
          };
          uint32_t mask[kBlocks], cmask[kBlocks];
          int total = 0;
#pragma unroll
          for (int bk = 0; bk < kBlocks; ++bk) {
            const int col0 = h * kSeg + part * Cfg<kQ>::kPartCols + bk * 32;
            mask[bk] = 0u;
            cmask[bk] = 0u;
            if (n0 + col0 < Q.N) {  // uniform
              uint32_t v[32];
              tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * kSeg + col0), v);
              tmem_ld_wait();
              const int nv = min(32, Q.N - (n0 + col0));
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (j < nv && __uint_as_float(v[j]) >= tau) mask[bk] |= 1u << j;
              total += __popc(mask[bk]);
              if (tr) {
                // lane l: which of the warp's 32 rows reach column l's threshold
                stage_block(v);
                const float tau_c = lane < nv ? Q.tau[Q.col_off + n0 + col0 + lane] : INFINITY;
                uint32_t cm = 0u;
#pragma unroll 8
                for (int r = 0; r < 32; ++r)
                  if (col_value(r) >= tau_c && row0 + r < Q.M) cm |= 1u << r;
                cmask[bk] = cm;
                __syncwarp();  // read before the next block is staged
              }
            }
          }
          int slot = 0;
          if (total > 0) slot = atomicAdd(Q.cnt + i_abs, total);
          int cbase[kBlocks];
#pragma unroll
          for (int bk = 0; bk < kBlocks; ++bk) {
            cbase[bk] = 0;
            if (cmask[bk] != 0u)
              cbase[bk] = atomicAdd(Q.cnt + Q.col_off + n0 + h * kSeg + part * Cfg<kQ>::kPartCols + bk * 32 + lane,
                                    __popc(cmask[bk]));
          }
          uint2* dst = Q.cand + (size_t)i_abs * Q.cap;
#pragma unroll
          for (int bk = 0; bk < kBlocks; ++bk) {
            if (__any_sync(0xffffffffu, (mask[bk] | cmask[bk]) != 0u)) {  // the TMEM load is warp-wide
              const int col0 = h * kSeg + part * Cfg<kQ>::kPartCols + bk * 32;
              const int j_abs0 = Q.col_off + n0 + col0;
              uint32_t v[32];
              tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * kSeg + col0), v);
              tmem_ld_wait();
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                if ((mask[bk] >> j) & 1u) {
                  if (slot < Q.cap) dst[slot] = make_uint2(ord_key(__uint_as_float(v[j])), (uint32_t)(j_abs0 + j));
                  ++slot;
                }
              }
              if (tr && __any_sync(0xffffffffu, cmask[bk] != 0u)) {
                // lane l writes column l's hits from the staged block
                stage_block(v);
                uint32_t m = cmask[bk];
                int sl = cbase[bk];
                uint2* cd = Q.cand + (size_t)(j_abs0 + lane) * Q.cap;
                while (m != 0u) {
                  const int r = __ffs(m) - 1;
                  m &= m - 1u;
                  if (sl < Q.cap) cd[sl] = make_uint2(ord_key(col_value(r)), (uint32_t)(Q.row_off + row0 + r));
                  ++sl;
                }
                __syncwarp();  // read before the next block is staged
              }
            }
          }
        }
        // bf16 output of a whole contraction: the warp's 128 columns of the segment are read and
        // rounded to bf16 in registers first, and the segment is released to the next tile's MMAs at
        // once; the staging and the stores follow (the MMAs of the next tile no longer wait for them)
        if (!kQ && !kF32 && Q.splits == 1 && Cfg<kQ>::kPartCols == 128) {
          const int c00 = h * kSeg + part * Cfg<kQ>::kPartCols;  // tile column of the warp's first block
          const uint32_t ta = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * kSeg + c00);
          uint32_t pk[2][32];  // [block][bf16 pair]: 64 columns per block
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            uint32_t v[32], w[32];
            tmem_ld_32x32b_x32(ta + (uint32_t)(64 * u), v);
            tmem_ld_32x32b_x32(ta + (uint32_t)(64 * u) + 32u, w);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              pk[u][e] = pack_bf16x2(__uint_as_float(v[2 * e]), __uint_as_float(v[2 * e + 1]));
              pk[u][16 + e] = pack_bf16x2(__uint_as_float(w[2 * e]), __uint_as_float(w[2 * e + 1]));
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(tempty_pl + (uint32_t)(buf + h) * 8u);
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int col0 = c00 + 64 * u;
            if (n0 + col0 >= Q.N || row0 >= Q.M) break;  // uniform across the warp
            if (lane == 0) bulk_wait_read0();            // the previous store has read the staging block
            __syncwarp();
            const uint32_t rbase = stg + (uint32_t)lane * 128u;
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const uint32_t dst = rbase + (uint32_t)(((k ^ (lane & 7)) & 7) << 4);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(pk[u][4 * k]),
                           "r"(pk[u][4 * k + 1]), "r"(pk[u][4 * k + 2]), "r"(pk[u][4 * k + 3])
                           : "memory");
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              tma_store_2d(&b.tmOut[p], stg, n0 + col0, row_st);
              bulk_commit();
            }
          }
          continue;
        }
        for (int cc = 0; !app && cc < Cfg<kQ>::kPartCols; cc += block_cols) {
          const int col0 = h * kSeg + part * Cfg<kQ>::kPartCols + cc;  // tile column of this block
          if (n0 + col0 >= Q.N || row0 >= Q.M) break;     // uniform across the warp
          const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * kSeg + col0);
          uint32_t v[32], w[32];
          tmem_ld_32x32b_x32(taddr, v);
          if (!f32) tmem_ld_32x32b_x32(taddr + 32u, w);
          tmem_ld_wait();
          if (lse_on) {
            const int nv = min(32, Q.N - (n0 + col0));  // valid columns of the block, >= 1
            float bm = __uint_as_float(v[0]);
#pragma unroll
            for (int j = 1; j < 32; ++j)
              if (j < nv) bm = fmaxf(bm, __uint_as_float(v[j]));
            const float mn = fmaxf(lm, bm);
            float acc = ls * __expf(lm - mn);
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (j < nv) acc += __expf(__uint_as_float(v[j]) - mn);
            lm = mn;
            ls = acc;
          }
          // the previous block's store must have read the staging buffer
          if (lane == 0) bulk_wait_read0();
          __syncwarp();
          // row `lane` of the block: 8 chunks of 16 B, chunk k at k ^ (row mod 8) (128-byte swizzle)
          const uint32_t rbase = stg + (uint32_t)lane * 128u;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            uint32_t a, b2, c2, d2;
            if (f32) {
              a = v[4 * k];
              b2 = v[4 * k + 1];
              c2 = v[4 * k + 2];
              d2 = v[4 * k + 3];
            } else {
              const uint32_t* src = k < 4 ? &v[k * 8] : &w[(k - 4) * 8];
              a = pack_bf16x2(__uint_as_float(src[0]), __uint_as_float(src[1]));
              b2 = pack_bf16x2(__uint_as_float(src[2]), __uint_as_float(src[3]));
              c2 = pack_bf16x2(__uint_as_float(src[4]), __uint_as_float(src[5]));
              d2 = pack_bf16x2(__uint_as_float(src[6]), __uint_as_float(src[7]));
            }
            const uint32_t dst = rbase + (uint32_t)(((k ^ (lane & 7)) & 7) << 4);
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(a), "r"(b2), "r"(c2), "r"(d2)
                         : "memory");
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&b.tmOut[p], stg, n0 + col0, row_st);
            bulk_commit();
          }
        }
        if (lse_on) {
          const int gc = n0 + h * kSeg + part * Cfg<kQ>::kPartCols;  // first column of the group
          if (gc < Q.N && row0 + lane < Q.M)
            Q.lse[(long long)(row0 + lane) * Q.ld_lse + gc / Cfg<kQ>::kPartCols] = make_float2(lm, ls);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(tempty_pl + (uint32_t)(buf + h) * 8u);
      }
      if (!ok) break;
    }
    // the output must be written before the CTA exits
    if (lane == 0) bulk_wait0();
  } else if (kQ && warp < 2 + kEpi + kConvWarps) {
    // ------------------------------------------------------------ weight dequantizers (both CTAs)
    const int cw = warp - 2 - kEpi;
    const int ct = cw * 32 + lane;
    const uint32_t wfull_pl = mapa_shared(smem_u32(&ctl->wfull[0]), 0);  // adapter-block TMA completions
    int qs = 0;          // code slot of the next main block
    uint32_t qpar = 0;   // its qfull parity
    uint32_t wseq = 0;   // contraction blocks so far: weight tile wseq % kWStages
    for (int it = 0;; ++it) {
      const int slot = it % kTileRing;
      bool got = mbar_wait_cluster(smem_u32(&ctl->tile_full[slot]), (uint32_t)((it / kTileRing) & 1), wc, abort_flag);
      got = __all_sync(0xffffffffu, got);
      if (!got) break;
      const int t = *reinterpret_cast<volatile int*>(&ctl->tile_id[slot]);
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(tile_empty_root + (uint32_t)slot * 8u);
      if (t < 0) break;
      int p, m0, n0, ks, kb0, kb1;
      decode_tile(b, t, p, m0, n0, ks, kb0, kb1);
      const GemmProblem& Q = b.prob[p];
      auto box_ok = [&](int h, int cc, int j) { return n0 + h * kSeg + cc * kHalf + j * 64 < Q.N; };
      bool ok = true;
      for (int kb = kb0; kb < kb1; ++kb) {
        const bool main = kb < Q.kb_main;
        const int wt = (int)(wseq % kWStages);
        // the weight tile's previous contents are consumed by the MMAs
        ok = mbar_wait_cluster(smem_u32(&ctl->wempty[wt]), ((wseq / kWStages) & 1u) ^ 1u, wc, abort_flag);
        if (ok && main) ok = mbar_wait(smem_u32(&ctl->qfull[qs]), qpar, wc, abort_flag);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) break;
        const uint32_t wdst = Cfg<kQ>::w_tile(base, wt);
        if (main) {
          dequant_stage<kBMn>(Cfg<kQ>::q_slot(base, qs), wdst, ct, c, n0, kb, Q.N);
          fence_proxy_async_smem();  // the tensor core reads what these threads wrote
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(smem_u32(&ctl->qempty[qs]));  // the code slot may be refilled
            mbar_arrive(smem_u32(&ctl->convd[wt]));
          }
          if (++qs == kQStages) {
            qs = 0;
            qpar ^= 1u;
          }
        } else {
          // adapter block: the bf16 rank-side boxes go straight into the weight tile by TMA
          if (cw == 0 && lane == 0) {
            const int kc = (kb - Q.kb_main) * kBK;
            const uint32_t bar = wfull_pl + (uint32_t)wt * 8u;
            if (c == 0) {
              // before this CTA's relay can arrive: the phase cannot complete without these bytes
              uint32_t boxes = 0;
              for (int h = 0; h < 2; ++h)
                for (int cc = 0; cc < 2; ++cc)
                  for (int j = 0; j < 2; ++j) boxes += box_ok(h, cc, j) ? 1u : 0u;
              mbar_expect_tx(smem_u32(&ctl->wfull[wt]), kBox * boxes);
            }
            for (int h = 0; h < 2; ++h) {
              for (int j = 0; j < 2; ++j) {
                if (!box_ok(h, c, j)) continue;
                const int col = n0 + h * kSeg + c * kHalf + j * 64;
                tma_load_2d_pair(wdst + h * kBSeg + j * kBox, &b.tmB2[p], bar, kBMn ? col : kc, kBMn ? kc : col);
              }
            }
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(smem_u32(&ctl->convd[wt]));
        }
        ++wseq;
      }
      if (!ok) break;
    }
  } else if (kQ && warp == 2 + kEpi + kConvWarps + 1) {
    // ------------------------------------------------------------ relay (both CTAs)
    if (lane == 0) {
      const uint32_t wfull_pl = mapa_shared(smem_u32(&ctl->wfull[0]), 0);
      uint32_t wseq = 0;
      for (int it = 0;; ++it) {
        const int slot = it % kTileRing;
        if (!mbar_wait_cluster(smem_u32(&ctl->tile_full[slot]), (uint32_t)((it / kTileRing) & 1), wc, abort_flag))
          break;
        const int t = *reinterpret_cast<volatile int*>(&ctl->tile_id[slot]);
        mbar_arrive_cluster(tile_empty_root + (uint32_t)slot * 8u);
        if (t < 0) break;
        int p, m0, n0, ks, kb0, kb1;
        decode_tile(b, t, p, m0, n0, ks, kb0, kb1);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb, ++wseq) {
          const int wt = (int)(wseq % kWStages);
          if (!mbar_wait(smem_u32(&ctl->convd[wt]), (wseq / kWStages) & 1u, wc, abort_flag)) {
            ok = false;
            break;
          }
          // cumulative release: covers the dequantizing warps' writes this thread acquired
          mbar_arrive_cluster(wfull_pl + (uint32_t)wt * 8u);
        }
        if (!ok) break;
      }
    }
  } else if (kQ) {
    // ------------------------------------------------------------ code producer (both CTAs)
    if (lane == 0) {
      int qs = 0;
      uint32_t qpar = 0;
      int qfills = 0;
      for (int it = 0;; ++it) {
        const int slot = it % kTileRing;
        if (!mbar_wait_cluster(smem_u32(&ctl->tile_full[slot]), (uint32_t)((it / kTileRing) & 1), wc, abort_flag))
          break;
        const int t = *reinterpret_cast<volatile int*>(&ctl->tile_id[slot]);
        mbar_arrive_cluster(tile_empty_root + (uint32_t)slot * 8u);
        if (t < 0) break;
        int p, m0, n0, ks, kb0, kb1;
        decode_tile(b, t, p, m0, n0, ks, kb0, kb1);
        const GemmProblem& Q = b.prob[p];
        auto box_ok = [&](int h, int j) { return n0 + h * kSeg + c * kHalf + j * 64 < Q.N; };
        // bytes of this CTA's code and (s, b) boxes per block
        uint32_t tx_q = 0;
        for (int h = 0; h < 2; ++h) {
          if (kBMn) {
            tx_q += box_ok(h, 0) ? 4096u + 1024u : 0u;
          } else {
            tx_q += box_ok(h, 0) ? 2048u : 0u;
            for (int j = 0; j < 2; ++j) tx_q += box_ok(h, j) ? 2048u : 0u;
          }
        }
        bool ok = true;
        for (int kb = kb0; kb < min(kb1, Q.kb_main); ++kb) {
          if (!mbar_wait(smem_u32(&ctl->qempty[qs]), qpar ^ 1u, wc, abort_flag)) {
            ok = false;
            break;
          }
          const uint32_t qbar = smem_u32(&ctl->qfull[qs]);
          const uint32_t codes = Cfg<kQ>::q_slot(base, qs);
          const uint32_t params = codes + kQCodes;
          mbar_arrive_expect_tx(qbar, tx_q);
          ++qfills;
          for (int h = 0; h < 2; ++h) {
            const int colh = n0 + h * kSeg + c * kHalf;
            if (!box_ok(h, 0)) continue;
            if (kBMn) {
              // W rows 64 kb ..; this CTA's 128 output columns = 64 code bytes, 2 groups
              tma_load_2d(codes + h * 4096, &b.tmQ[p], qbar, colh / 2, kb * kBK);
              tma_load_2d(params + h * 1024, &b.tmP[p], qbar, ((colh >> 6) & ~3) * 2, kb * kBK);
            } else {
              for (int j = 0; j < 2; ++j)
                if (box_ok(h, j)) tma_load_2d(codes + (h * 2 + j) * 2048, &b.tmQ[p], qbar, kb * 32, colh + j * 64);
              tma_load_2d(params + h * 2048, &b.tmP[p], qbar, (kb & ~3) * 2, colh);
            }
          }
          if (++qs == kQStages) {
            qs = 0;
            qpar ^= 1u;
          }
        }
        if (!ok) break;
      }
      ctl->qfills = qfills;
    }
  }

  if constexpr (kCS) {
    // ------------------------------------------------------------ cluster split: sum the two halves
    // After the cluster barrier both pairs' contractions are complete, so every CTA's ring is idle:
    // its first 64 KB receive the other pair's values for this CTA's rows and this pair's 128 columns,
    // the next 64 KB stage the values this CTA sends.  Layout of both: 128 rows x 128 fp32 columns,
    // 16-byte chunk kc of row r at chunk kc ^ (r mod 8) (a warp's 32 rows hit every bank group once).
    // The warps over the other pair's columns stage their rows and send them with one bulk copy per
    // warp (16 KB) to the same-position CTA of the other pair, completing on its barrier `xchg`; the
    // warps over this pair's columns wait for the 64 KB to arrive, add them (fp32, two terms: the same
    // sum whichever pair adds), round to bf16 and store.
    cluster_sync_all();
    if (warp >= 2 && warp < 2 + kEpi && !*abort_flag) {
      int p, m0, n0, ks, kb0, kb1;
      decode_tile<kTileN>(b, cs_tile, p, m0, n0, ks, kb0, kb1, cs_half);
      const GemmProblem& Q = b.prob[p];
      const int q = warp & 3, part = (warp - 2) >> 2;
      const uint32_t row = (uint32_t)(q * 32 + lane);
      const uint32_t tl = tmem_base + ((uint32_t)(q * 32) << 16);
      constexpr uint32_t kRecv = 0, kSend = 128u * 512u;  // offsets in the ring
      auto chunk = [&](uint32_t kc) { return row * 512u + (((kc ^ row) & 7u) | (kc & ~7u)) * 16u; };
      if (part != cs_half) {
        for (int blk = 0; blk < 4; ++blk) {
          uint32_t v[32];
          tmem_ld_32x32b_x32(tl + (uint32_t)(part * kHalf + blk * 32), v);
          tmem_ld_wait();
#pragma unroll
          for (int k = 0; k < 8; ++k)
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(base + kSend + chunk((uint32_t)(blk * 8 + k))),
                         "r"(v[4 * k]), "r"(v[4 * k + 1]), "r"(v[4 * k + 2]), "r"(v[4 * k + 3])
                         : "memory");
        }
        fence_proxy_async_smem();  // the bulk copy reads what these threads wrote
        __syncwarp();
        if (lane == 0) {
          const uint32_t peer = crank ^ 2u;  // the same position in the other pair
          const uint32_t rows = (uint32_t)(q * 32) * 512u;
          bulk_copy_to_peer(mapa_shared(base + kRecv + rows, peer), base + kSend + rows, 32u * 512u,
                            mapa_shared(smem_u32(&ctl->xchg), peer));
        }
      } else {
        if (q == 0 && lane == 0) mbar_arrive_expect_tx(smem_u32(&ctl->xchg), 128u * 512u);
        bool got = mbar_wait(smem_u32(&ctl->xchg), 0u, wc, abort_flag);
        got = __all_sync(0xffffffffu, got);
        const int row0 = m0 + c * kHalf + q * 32;
        const uint32_t stg = epi_base + (uint32_t)(warp - 2) * kEpiStage;
        for (int u = 0; got && u < 2; ++u) {
          const int col = part * kHalf + u * 64;
          if (n0 + col >= Q.N || row0 >= Q.M) break;  // uniform
          uint32_t v[32], w[32];
          tmem_ld_32x32b_x32(tl + (uint32_t)col, v);
          tmem_ld_32x32b_x32(tl + (uint32_t)col + 32u, w);
          tmem_ld_wait();
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            uint32_t o[4];
            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(o[0]), "=r"(o[1]), "=r"(o[2]), "=r"(o[3])
                         : "r"(base + kRecv + chunk((uint32_t)(u * 16 + k)))
                         : "memory");
            uint32_t* d = k < 8 ? &v[4 * k] : &w[4 * (k - 8)];
#pragma unroll
            for (int e = 0; e < 4; ++e) d[e] = __float_as_uint(__uint_as_float(d[e]) + __uint_as_float(o[e]));
          }
          if (lane == 0) bulk_wait_read0();  // the previous store has read the staging block
          __syncwarp();
          const uint32_t rbase = stg + (uint32_t)lane * 128u;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const uint32_t* src = k < 4 ? &v[k * 8] : &w[(k - 4) * 8];
            const uint32_t a = pack_bf16x2(__uint_as_float(src[0]), __uint_as_float(src[1]));
            const uint32_t b2 = pack_bf16x2(__uint_as_float(src[2]), __uint_as_float(src[3]));
            const uint32_t c2 = pack_bf16x2(__uint_as_float(src[4]), __uint_as_float(src[5]));
            const uint32_t d2 = pack_bf16x2(__uint_as_float(src[6]), __uint_as_float(src[7]));
            const uint32_t dst = rbase + (uint32_t)(((k ^ (lane & 7)) & 7) << 4);
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(dst), "r"(a), "r"(b2), "r"(c2), "r"(d2)
                         : "memory");
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&b.tmOut[p], stg, n0 + col, row0);
            bulk_commit();
          }
        }
        if (lane == 0) bulk_wait0();
      }
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) {
    // every MMA of the pair has finished before tensor memory is released
    if (!mbar_wait_drain(smem_u32(&ctl->drain), 0, b.limit_ns > kDrainNs ? b.limit_ns : kDrainNs))
      atomicCAS(b.status, 0, kStatusTimeout);
    if (*abort_flag) {
      // A wait gave up, so copies may still be in flight into this CTA's ring.  The barriers
      // armed here track them: wait (bounded, kAbortDrainNs each) until the last fill of every
      // ring stage (even CTA: both CTAs' operand boxes) and of every code slot (4-bit) has
      // landed.  Copies that signal the peer's barriers, or that were issued for a fill that was
      // never armed, are not observable here: a fixed 50 us margin follows for those.
      const int nf = ctl->fills, nq = ctl->qfills;
      if (c == 0)
        for (int i = nf - 1; i >= 0 && i >= nf - kStages; --i)
          if (!mbar_wait_drain(smem_u32(&ctl->full[i % kStages]), (uint32_t)((i / kStages) & 1), kAbortDrainNs))
            atomicCAS(b.status, 0, kStatusTimeout);
      if (kQ)
        for (int i = nq - 1; i >= 0 && i >= nq - kQStages; --i)
          if (!mbar_wait_drain(smem_u32(&ctl->qfull[i % kQStages]), (uint32_t)((i / kQStages) & 1), kAbortDrainNs))
            atomicCAS(b.status, 0, kStatusTimeout);
      const uint64_t t0 = global_timer_ns();
      while (global_timer_ns() - t0 < 50000ull) {
      }
    }
  }
  // with early inputs a CTA may have loaded no adapter slab: it still leaves only after the previous
  // grid, so that this grid's completion implies that grid's (the next grid waits for this one only)
  if (b.early_inputs && threadIdx.x == 0) griddep_wait();
  __syncthreads();
  cluster_sync_all();  // no cross-CTA access is pending in either CTA
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
}

constexpr int kLseGroup = 128;  // columns of one log-sum-exp partial
static_assert(kLseGroup == Cfg<false>::kPartCols, "the epilogue's column group");

// Threads the split reduce runs for a problem, a multiple of 32: one per 4
// consecutive columns of a row; with log-sum-exp partials one warp per
// (row, 128-column group).
__host__ __device__ inline long long reduce_items(const GemmProblem& Q) {
  if (Q.splits <= 1) return 0;
  const long long n = Q.lse ? (long long)Q.M * ((Q.N + kLseGroup - 1) / kLseGroup) * 32
                            : (long long)Q.M * ((Q.N + 3) / 4);
  return (n + 31) / 32 * 32;
}

__device__ __forceinline__ void lse_merge2(float& m, float& s, float m2, float s2) {
  if (m2 > m) {
    s = s * __expf(m - m2) + s2;
    m = m2;
  } else if (m2 > -INFINITY) {
    s += s2 * __expf(m2 - m);
  }
}

// out[m, n] = sum over s of part[s * m_pad + m, n], s in order, 4 columns per
// thread; for a problem with lse partials also each (row, column group)'s
// (max, sum of exp) over the summed values, one warp per group.
__global__ void __launch_bounds__(256) split_reduce_kernel(const __grid_constant__ GemmBatch b, long long total) {
  griddep_wait();
  griddep_launch_dependents();
  long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x;
  if (e >= total) return;  // total is a multiple of 32: whole warps leave
  int p = 0;
  for (; p < b.num_problems; ++p) {
    const long long per = reduce_items(b.prob[p]);
    if (e < per) break;
    e -= per;
  }
  const GemmProblem& Q = b.prob[p];
  int m, n;
  if (Q.lse) {
    const int ng = (Q.N + kLseGroup - 1) / kLseGroup;
    const long long w = e >> 5;
    m = (int)(w / ng);
    n = (int)(w % ng) * kLseGroup + (int)(e & 31) * 4;
  } else {
    const int n4 = (Q.N + 3) / 4;
    m = (int)(e / n4);
    n = (int)(e % n4) * 4;
  }
  const bool row_ok = m < Q.M;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  if (row_ok && n < Q.N) {
    for (int s = 0; s < Q.splits; ++s) {
      const float* src = Q.part + ((size_t)s * Q.m_pad + m) * Q.ldp + n;
      if (n + 3 < Q.N) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(src));
        acc[0] += v.x;
        acc[1] += v.y;
        acc[2] += v.z;
        acc[3] += v.w;
      } else {
        for (int q = 0; q < 4 && n + q < Q.N; ++q) acc[q] += src[q];
      }
    }
    for (int q = 0; q < 4 && n + q < Q.N; ++q) {
      if (Q.out_f32)
        static_cast<float*>(Q.out)[(size_t)m * Q.ldo + n + q] = acc[q];
      else
        static_cast<__nv_bfloat16*>(Q.out)[(size_t)m * Q.ldo + n + q] = __float2bfloat16_rn(acc[q]);
    }
  }
  if (Q.lse) {  // warp-uniform
    float lm = -INFINITY, ls = 0.f;
    for (int q = 0; q < 4; ++q)
      if (row_ok && n + q < Q.N) lse_merge2(lm, ls, acc[q], 1.f);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, lm, o), s2 = __shfl_xor_sync(0xffffffffu, ls, o);
      lse_merge2(lm, ls, m2, s2);
    }
    if ((e & 31) == 0 && row_ok) Q.lse[(size_t)m * Q.ld_lse + n / kLseGroup] = make_float2(lm, ls);
  }
}

}  // namespace

cudaError_t launch_split_reduce(const GemmBatch& batch, cudaStream_t stream) {
  long long total = 0;
  for (int p = 0; p < batch.num_problems; ++p) total += reduce_items(batch.prob[p]);
  if (total == 0) return cudaSuccess;
  return launch_kernel(split_reduce_kernel, dim3((unsigned)((total + 255) / 256)), dim3(256), 0, stream, 1, batch,
                       total);
}

size_t fused_gemm_smem_bytes() { return smem_bytes<false>(); }

template <bool kBMn, bool kQ, bool kF32, bool kCS = false>
cudaError_t launch_variant(const GemmBatch& batch, int pairs, cudaStream_t stream) {
  constexpr size_t smem = smem_bytes<kQ>();
  static std::atomic<unsigned long long> attr_done{0};
  const cudaError_t e = set_smem_once(fused_lora_gemm<kBMn, kQ, kF32, kCS>, (int)smem, attr_done);
  if (e != cudaSuccess) return e;
  // kCS: one tile per cluster of two pairs; otherwise persistent pairs
  const unsigned grid = kCS ? (unsigned)(4 * batch.total_tiles) : (unsigned)(2 * pairs);
  return launch_kernel(fused_lora_gemm<kBMn, kQ, kF32, kCS>, dim3(grid), dim3(Cfg<kQ>::kThreads), smem, stream,
                       kCS ? 4 : 2, batch);
}

// Clusters of four of the cluster-split kernel that can run at once on this
// device (0 if the query fails), cached per device and majorness.
template <bool kBMn>
int cs_max_clusters() {
  static std::atomic<int> cache[64][1];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  int v = cache[dev][0].load(std::memory_order_acquire);
  if (v != 0) return v > 0 ? v : 0;
  constexpr size_t smem = smem_bytes<false>();
  static std::atomic<unsigned long long> attr_done{0};
  int n = -1;
  if (set_smem_once(fused_lora_gemm<kBMn, false, false, true>, (int)smem, attr_done) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(4 * 64);
    cfg.blockDim = dim3(Cfg<false>::kThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 4;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int k = 0;
    if (cudaOccupancyMaxActiveClusters(&k, fused_lora_gemm<kBMn, false, false, true>, &cfg) == cudaSuccess && k > 0)
      n = k;
    else
      cudaGetLastError();
  }
  cache[dev][0].store(n, std::memory_order_release);
  return n > 0 ? n : 0;
}

int gemm_cs_max_clusters(bool b_mn_major) {
  return b_mn_major ? cs_max_clusters<true>() : cs_max_clusters<false>();
}

cudaError_t launch_fused_gemm_cs(const GemmBatch& batch, bool b_mn_major, cudaStream_t stream) {
  if (batch.total_tiles <= 0) return cudaSuccess;
  return b_mn_major ? launch_variant<true, false, false, true>(batch, 0, stream)
                    : launch_variant<false, false, false, true>(batch, 0, stream);
}

cudaError_t launch_fused_gemm(const GemmBatch& batch, bool b_mn_major, bool q4, int num_sms, cudaStream_t stream,
                              bool f32_out) {
  if (batch.total_tiles <= 0) return cudaSuccess;
  const int pairs = batch.total_tiles < num_sms / 2 ? batch.total_tiles : num_sms / 2;
  if (f32_out) {
    if (b_mn_major || q4) return cudaErrorInvalidValue;  // only the plain forward form writes fp32
    return launch_variant<false, false, true>(batch, pairs, stream);
  }
  if (q4)
    return b_mn_major ? launch_variant<true, true, false>(batch, pairs, stream)
                      : launch_variant<false, true, false>(batch, pairs, stream);
  return b_mn_major ? launch_variant<true, false, false>(batch, pairs, stream)
                    : launch_variant<false, false, false>(batch, pairs, stream);
}

int gemm_tile_m() { return kBM; }
int gemm_lse_group() { return kLseGroup; }
int gemm_tile_n() { return kBN; }
int gemm_tile_n_f32() { return kSeg; }
int gemm_tile_k() { return kBK; }

}  // namespace lora
