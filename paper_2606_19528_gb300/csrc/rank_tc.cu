// Rank-r products of the LoRA linear on the 5th-generation tensor cores.
// Row products, out[t, j] = scale * sum_c X[t, c] * W[j, c]:
//   su = s x A^T      (forward; x [T, K], A [r, K])
//   sv = s dy B       (backward, r > 16; dy [T, N], B given transposed, B^T [r, N])
// Column products, out[c, j] = sum_t X[t, c] * S[t, j] (S given transposed):
//   dB = dy^T su      (backward, r > 16; dy [T, N], su^T [r, T])
//   dA = sv^T x       (x [T, K], sv^T [r, T])
// (Up to r = 16 the backward's sv and dB come from one fused pass over dy.)
// One problem per activation X, with the rank side the concatenation of
// every projection reading X (q, k and v share x).  Each is a skinny
// contraction that streams the tall X once: an output tile is 128 rows of X's
// long side (tokens for a row product, columns for a column product) by the
// padded rank, reduced over 64-wide chunks of the other side.  The MMA is
// M = 128 x N = rank x K = 16 with A = the X tile (K-major for row products;
// MN-major, straight from X's row-major layout, for column products) and B =
// the rank-side tile (always K-major).
// Per CTA (persistent, one per SM): warp 0 streams X tiles (16 KB) and the
// matching rank-side tiles by TMA into a deep ring of shared-memory stages;
// one thread of warp 1 issues tcgen05.mma into a TMEM accumulator; warps 2..5
// read the accumulator back (one output row per thread) and write the
// outputs, or fp32 partials when a tile's reduction spans several work units
// (summed in unit order by a second pass, so results never depend on
// scheduling).  Two accumulators let the read-back of one unit overlap the
// next unit's loads and MMAs.  The MMAs are tiny (N = rank), and a stream of
// them from one thread takes ~47 cycles per MMA whatever N up to 64; one CTA
// streams X at ~45-60 GB/s, bounded by the X bytes its ring keeps in flight
// (16 KB boxes, 8 stages) against the load latency, so these kernels fill the
// HBM bandwidth only on many SMs.  Every wait is bounded.
#include "rank_store.cuh"

namespace lora {

namespace {

constexpr int kRows = 128;                        // output rows per tile = TMEM lanes
constexpr int kChunk = 64;                        // reduction length per stage
constexpr uint32_t kXBytes = kRows * kChunk * 2;  // 16 KB
constexpr uint32_t kXHalf = kXBytes / 2;          // one 64 x 64 box of a column product
constexpr int kThreads = 192;
constexpr long long kDrainNs = 1000000000ll;

template <int R>
struct TcRing {
  static constexpr uint32_t kStageBytes = (kXBytes + 128u * R + 1023u) & ~1023u;
  static constexpr int kStages = (int)(196608u / kStageBytes) < 12 ? (int)(196608u / kStageBytes) : 12;
  static constexpr uint32_t kTmemCols = 2 * R <= 32 ? 32 : 2 * R;  // two accumulators, power of two
};

struct __align__(8) TcCtl {
  uint64_t full[12];
  uint64_t empty[12];
  uint64_t tfull[2];
  uint64_t tempty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

template <int R>
constexpr size_t tc_smem_bytes() {
  return 1024 + (size_t)TcRing<R>::kStages * TcRing<R>::kStageBytes + sizeof(TcCtl);
}

// What differs between the row and the column products.
template <bool kCol>
struct Side;
template <>
struct Side<false> {
  using Batch = RowBatch;
  using Prob = RowProb;
  __device__ static int rows(const Prob& P) { return P.T; }
  __device__ static int red(const Prob& P) { return P.C; }
  __device__ static int rank(const Prob& P, int k) { return P.rw[k]; }
  __device__ static const CUtensorMap* rmap(const Prob& P, int k) { return &P.tmW[k]; }
};
template <>
struct Side<true> {
  using Batch = ColBatch;
  using Prob = ColProb;
  __device__ static int rows(const Prob& P) { return P.C; }
  __device__ static int red(const Prob& P) { return P.T; }
  __device__ static int rank(const Prob& P, int k) { return P.rs[k]; }
  __device__ static const CUtensorMap* rmap(const Prob& P, int k) { return &P.tmS[k]; }
};

template <typename Batch>
__device__ __forceinline__ void decode_unit(const Batch& b, int u, int& pi, int& tile, int& piece) {
  pi = 0;
  while (pi + 1 < b.n && u >= b.p[pi + 1].unit_begin) ++pi;
  const int lu = u - b.p[pi].unit_begin;
  tile = lu / b.p[pi].upt;
  piece = lu % b.p[pi].upt;
}

template <int R, bool kCol>
__global__ void __launch_bounds__(kThreads, 1) rank_mma_kernel(const __grid_constant__ typename Side<kCol>::Batch b) {
  using G = TcRing<R>;
  using S = Side<kCol>;
  using Prob = typename S::Prob;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  TcCtl* ctl = reinterpret_cast<TcCtl*>(smem_raw + (base - raw) + (size_t)G::kStages * G::kStageBytes);
  volatile int* abort_flag = &ctl->abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{b.status, b.limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < G::kStages; ++s) {
      mbar_init(smem_u32(&ctl->full[s]), 1);
      mbar_init(smem_u32(&ctl->empty[s]), 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(smem_u32(&ctl->tfull[a]), 1);
      mbar_init(smem_u32(&ctl->tempty[a]), 4);  // one arrival per epilogue warp
    }
    mbar_init(smem_u32(&ctl->drain), 1);
    ctl->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&ctl->tmem_base), G::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  griddep_wait();  // X and the rank sides may come from the previous grid
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
        int pi, tile, piece;
        decode_unit(b, u, pi, tile, piece);
        const Prob& P = b.p[pi];
        const int r0 = tile * kRows;
        const int k_begin = piece * b.unit_chunks * kChunk;
        const int nch = (min(S::red(P), k_begin + b.unit_chunks * kChunk) - k_begin + kChunk - 1) / kChunk;
        // a column tile whose second half lies past C loads only the first box
        const bool hi = !kCol || r0 + kChunk < S::rows(P);
        const uint32_t tx = (uint32_t)P.tx_bytes - (hi ? 0u : kXHalf);
        for (int ch = 0; ch < nch; ++ch) {
          if (!mbar_wait(smem_u32(&ctl->empty[stage]), phase ^ 1u, wc, abort_flag)) {
            ok = false;
            break;
          }
          const uint32_t full = smem_u32(&ctl->full[stage]);
          const uint32_t xs = base + (uint32_t)stage * G::kStageBytes;
          const int k0 = k_begin + ch * kChunk;
          mbar_arrive_expect_tx(full, tx);
          if constexpr (kCol) {
            // X^T as an MN-major operand: two 64-column x 64-token boxes
            tma_load_2d(xs, &P.tmX, full, r0, k0);
            if (hi) tma_load_2d(xs + kXHalf, &P.tmX, full, r0 + kChunk, k0);
          } else {
            tma_load_2d(xs, &P.tmX, full, k0, r0);
          }
          int off = 0;
          for (int k = 0; k < P.nblk; ++k) {
            tma_load_2d(xs + kXBytes + (uint32_t)off * 128u, S::rmap(P, k), full, k0, 0);
            off += pad8(S::rank(P, k));
          }
          ++issued;
          if (++stage == G::kStages) {
            stage = 0;
            phase ^= 1u;
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
      int it = 0;
      bool ok = true;
      // stage 0's operand descriptors: X (K-major rows, or MN-major with the boxes kXHalf apart)
      // and the rank side after it
      const uint64_t desc_a = kCol ? sw128_desc(base, kXHalf, 1024) : sw128_desc(base, 16, 1024);
      const uint64_t desc_b = sw128_desc(base + kXBytes, 16, 1024);
      for (int u = blockIdx.x; u < b.units && ok; u += gridDim.x, ++it) {
        int pi, tile, piece;
        decode_unit(b, u, pi, tile, piece);
        const Prob& P = b.p[pi];
        const int k_begin = piece * b.unit_chunks * kChunk;
        const int nch = (min(S::red(P), k_begin + b.unit_chunks * kChunk) - k_begin + kChunk - 1) / kChunk;
        const uint32_t idesc = idesc_bf16_f32(kRows, P.rpad, kCol ? 1 : 0, 0);
        const int acc = it & 1;
        if (!mbar_wait(smem_u32(&ctl->tempty[acc]), (uint32_t)(((it >> 1) & 1) ^ 1), wc, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(acc * R);
        for (int ch = 0; ch < nch; ++ch) {
          if (!mbar_wait(smem_u32(&ctl->full[stage]), phase, wc, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // this stage's descriptors: stage 0's with the start address moved (addr >> 4 in the
          // low 14 bits of the descriptor; shared-memory offsets never carry out of them)
          const uint32_t soff = (uint32_t)stage * (G::kStageBytes >> 4);
          const uint64_t ad = desc_a + soff, bd = desc_b + soff;
#pragma unroll
          for (int k = 0; k < kChunk / 16; ++k) {
            // MN-major A: 16 reduction rows of 128 B per step, the two 64-wide boxes 8 KB apart
            umma_bf16(d_tmem, ad + (uint32_t)(kCol ? k * 128 : k * 2), bd + (uint32_t)(k * 2), idesc,
                      (ch | k) != 0 ? 1u : 0u);
          }
          issued_any = true;
          umma_commit(smem_u32(&ctl->empty[stage]));
          if (++stage == G::kStages) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(smem_u32(&ctl->tfull[acc]));
      }
    }
  } else {
    // ---------------------------------------------------------------- epilogue
    const int q = warp & 3;  // TMEM lane quadrant: output rows q*32 .. q*32+31
    int it = 0;
    for (int u = blockIdx.x; u < b.units; u += gridDim.x, ++it) {
      int pi, tile, piece;
      decode_unit(b, u, pi, tile, piece);
      const Prob& P = b.p[pi];
      const int acc = it & 1;
      // no group barrier follows, so each warp may leave on its own
      if (!mbar_wait(smem_u32(&ctl->tfull[acc]), (uint32_t)((it >> 1) & 1), wc, abort_flag)) break;
      tc_fence_after();
      const int row = q * 32 + lane;
      const int g = tile * kRows + row;
      const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * R);
      float* part = P.upt > 1 ? b.partials + P.part_off + ((size_t)(tile * P.upt + piece) * kRows + row) * P.rpad
                              : nullptr;
#pragma unroll
      for (int j0 = 0; j0 < R; j0 += 16) {
        if (j0 < P.rpad) {  // uniform across the warp
          uint32_t v[16];
          tmem_ld_32x32b_x16(taddr + (uint32_t)j0, v);
          tmem_ld_wait();
          if (part != nullptr) {
#pragma unroll
            for (int e = 0; e < 16; e += 4)
              __stcg(reinterpret_cast<float4*>(part + j0 + e),
                     make_float4(__uint_as_float(v[e]), __uint_as_float(v[e + 1]), __uint_as_float(v[e + 2]),
                                 __uint_as_float(v[e + 3])));
          } else if (g < S::rows(P)) {
#pragma unroll
            for (int h = 0; h < 16; h += 8) {
              if (j0 + h < P.rpad) {
                if constexpr (kCol)
                  col_store8(P, g, j0 + h, v + h);
                else
                  row_store8(P, g, j0 + h, v + h);
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(smem_u32(&ctl->tempty[acc]));
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
    tmem_dealloc(tmem_base, G::kTmemCols);
  }
}

template <int R, bool kCol>
cudaError_t launch_r(const typename Side<kCol>::Batch& b, int ctas, cudaStream_t st) {
  constexpr int smem = (int)tc_smem_bytes<R>();
  static std::atomic<unsigned long long> attr_done{0};
  const cudaError_t e = set_smem_once(rank_mma_kernel<R, kCol>, smem, attr_done);
  if (e != cudaSuccess) return e;
  const int grid = b.units < ctas ? b.units : ctas;
  return launch_kernel(rank_mma_kernel<R, kCol>, dim3(grid), dim3(kThreads), smem, st, 1, b);
}

template <bool kCol>
cudaError_t launch_side(const typename Side<kCol>::Batch& b, int rmax, int ctas, cudaStream_t st) {
  if (b.n <= 0 || b.units <= 0 || ctas <= 0) return cudaSuccess;
  if (rmax <= 16) return launch_r<16, kCol>(b, ctas, st);
  if (rmax <= 32) return launch_r<32, kCol>(b, ctas, st);
  if (rmax <= 64) return launch_r<64, kCol>(b, ctas, st);
  return launch_r<128, kCol>(b, ctas, st);
}

}  // namespace

int rank_mma_tile() { return kRows; }

cudaError_t launch_rowmma(const RowBatch& b, int rmax, int ctas, cudaStream_t st) {
  cudaError_t e = launch_side<false>(b, rmax, ctas, st);
  if (e != cudaSuccess || b.red_total <= 0) return e;
  return launch_reduce_rows(b, st);
}

cudaError_t launch_colmma(const ColBatch& b, int rmax, int ctas, cudaStream_t st) {
  cudaError_t e = launch_side<true>(b, rmax, ctas, st);
  if (e != cudaSuccess || b.red_total <= 0) return e;
  return launch_reduce_cols(b, st);
}

}  // namespace lora
