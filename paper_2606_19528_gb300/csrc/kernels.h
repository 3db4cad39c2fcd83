// Internal interface between the C ABI (api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <atomic>

namespace lora {

// Counts one kernel launch (defined with the C ABI).
void note_launch();

// Whether kernels are launched with programmatic dependent launch (on unless
// the environment sets LORA_PDL=0).
bool pdl_enabled();

// Launches `kernel` on `st` with programmatic stream serialization (when
// enabled) and, for cluster_x > 1, clusters of cluster_x CTAs; counts it.
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                          int cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  unsigned n = 0;
  if (pdl_enabled()) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster_x > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = (unsigned)cluster_x;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
  note_launch();
  return e != cudaSuccess ? e : cudaGetLastError();
}

// Raises `kernel`'s dynamic shared-memory limit to `smem` bytes on the
// current device, once per device (the attribute belongs to the device's copy
// of the kernel); `done` is the kernel's bit set of devices already raised.
template <typename... KArgs>
cudaError_t set_smem_once(void (*kernel)(KArgs...), int smem, std::atomic<unsigned long long>& done) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned long long bit = 1ull << (dev & 63);
  if (done.load(std::memory_order_acquire) & bit) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess) done.fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

// ---------------------------------------------------------------- fused GEMM
constexpr int kMaxProblems = 8;

struct GemmProblem {
  void* out;           // [M, N] bf16 (fp32 when out_f32), leading dimension ldo
  int ldo;
  int out_f32;
  int M;               // tokens
  int N;               // output columns
  int Kmain;           // base contraction length
  int r;               // adapter slab length (rank)
  int num_n_tiles;     // tiles along N
  int tile_begin;      // first index of this problem in the batch's tile list
  int kb_main;         // contraction blocks of the base part
  int kb_total;        // base + adapter blocks
  int m_fast;          // 1: consecutive tiles walk M (the weight tile stays put)
  int num_m_tiles;
  // split contraction: splits > 1 cuts [0, kb_total) into ranges of kb_split
  // blocks; each (tile, split) writes an fp32 partial through tmOut, split s at
  // rows s * m_pad.., and split_reduce sums the splits in order into out
  int splits;
  int kb_split;
  int m_pad;           // num_m_tiles * tile rows
  float* part;         // partials [splits * m_pad, ldp]
  int ldp;
  // fp32 output without splits only: per row and 128-column group g, the
  // group's (max, sum of exp(z - max)) over columns < N, at lse[row * ld_lse + g]
  float2* lse;
  int ld_lse;
  // fp32 output without splits only, instead of storing the output: with
  // i = row_off + m and j = col_off + n the absolute indices of z[m, n],
  // z >= tau[i] is appended as (order key, j) to i's list cand[i * cap ..],
  // cnt[i] counting every hit (also past cap); with sym set, tiles with
  // n0 > 0 (off the diagonal block) also append (order key, i) to j's list
  // when z >= tau[j]
  const float* tau;
  int* cnt;
  uint2* cand;
  int cap;
  int row_off, col_off, sym;
};

// Rows of each problem of the symmetric top-k contraction: its columns start at
// the problem's first row, so tiles with n0 < kSymRows form the diagonal block.
constexpr int kSymRows = 512;

// One launch: up to kMaxProblems independent fused contractions.
//  tmA  [M, Kmain] K-major (x or dy)        tmA2 [M, r] K-major (su or sv)
//  forward:  tmB  W [N, Kmain] K-major       tmB2 B [N, r] K-major
//  backward: tmB  W [Kmain, N] MN-major      tmB2 A [r, N] MN-major
struct GemmBatch {
  CUtensorMap tmA[kMaxProblems];
  CUtensorMap tmA2[kMaxProblems];
  CUtensorMap tmB[kMaxProblems];
  CUtensorMap tmB2[kMaxProblems];
  CUtensorMap tmOut[kMaxProblems];  // out [M, N]: 128-byte rows of 32 rows (64 bf16 or 32 fp32), 128-byte swizzle
  // 4-bit weights only: codes [d_out, d_in / 2] bytes and (s, b) pairs [d_out, d_in / 64, 2] bf16
  CUtensorMap tmQ[kMaxProblems];
  CUtensorMap tmP[kMaxProblems];
  GemmProblem prob[kMaxProblems];
  int num_problems;
  int total_tiles;
  int* tile_counter;   // zero at launch; hands out tiles in list order
  int* status;
  long long limit_ns;
  // 1: an earlier kernel of the same call precedes this launch on its stream, so the call's inputs
  // (the base contraction's operands) were complete before this grid started and its main blocks may
  // be loaded before the previous grid ends; only the adapter slab's activations (su or sv) wait
  int early_inputs;
};

// b_mn_major: the weight operand is contracted over its rows (backward);
// q4: every problem's base weight is given as 4-bit codes (tmQ, tmP).
// f32_out (forward form, bf16 weights only): the output is fp32 (tmOut an fp32
// map with 32 x 32 boxes) instead of bf16.
cudaError_t launch_fused_gemm(const GemmBatch& batch, bool b_mn_major, bool q4, int num_sms, cudaStream_t stream,
                              bool f32_out = false);
size_t fused_gemm_smem_bytes();
// Cluster split (bf16 weights and output, either majorness): one 256 x 256
// tile per cluster of two CTA pairs, each pair contracting half of the tile's
// blocks, the halves summed through distributed shared memory.  The batch
// lists each tile once (num_n_tiles over gemm_tile_n_f32() columns, splits 1);
// the grid is 4 CTAs per tile, all resident at once when the tile count is at
// most gemm_cs_max_clusters().
cudaError_t launch_fused_gemm_cs(const GemmBatch& batch, bool b_mn_major, cudaStream_t stream);
int gemm_cs_max_clusters(bool b_mn_major);
// out = sum over s of the split partials, in split order, for every problem
// of the batch with splits > 1 (bf16 or fp32 per out_f32).
cudaError_t launch_split_reduce(const GemmBatch& batch, cudaStream_t stream);
int gemm_tile_m();
int gemm_tile_n_f32();  // tile columns of the fp32-output form (two accumulator buffers)
int gemm_lse_group();  // columns of one log-sum-exp partial
int gemm_tile_n();
int gemm_tile_k();

// ---------------------------------------------------------------- rank-r kernels
inline int rank_pad16(int r) { return (r + 15) / 16 * 16; }
inline int rank_pad8(int r) { return (r + 7) / 8 * 8; }

constexpr int kMaxRankBlocks = 4;     // projections fused into one problem
constexpr int kMaxRankProblems = 12;  // problems per launch

// Row product problem: out_b[t, j] = scale * sum_c X[t, c] * W_b[j, c] for
// every block b (one projection each) sharing the activation X [T, C]; W_b
// is [r_b, C] row-major (A of the adapter, or B of the adapter transposed).
// Blocks are concatenated at 8-aligned rank offsets; columns rw_b .. ld_out_b
// of out_b are written as zeros; out2_b (optional) gets columns < ld_out2_b
// and outT_b (optional) the transpose [pad8(r_b), T], zero rows past r_b.
struct RowProb {
  CUtensorMap tmX;                   // X [T, C]: box 64 columns x 128 tokens, 128-byte swizzle
  CUtensorMap tmW[kMaxRankBlocks];   // W_b [r_b, C]: box 64 columns x pad8(r_b) rows, 128-byte swizzle
  int T, C;
  int nblk;
  int rw[kMaxRankBlocks];
  __nv_bfloat16* out[kMaxRankBlocks];
  int ld_out[kMaxRankBlocks];
  __nv_bfloat16* out2[kMaxRankBlocks];
  int ld_out2[kMaxRankBlocks];
  __nv_bfloat16* outT[kMaxRankBlocks];
  float scale;
  int rpad;            // concatenated rank, rounded up to 16
  int tx_bytes;        // bytes one chunk stage receives (X box + rank-side boxes)
  int upt;             // work units per 128-token tile (each unit_chunks x 64 columns)
  int unit_begin;      // first unit of this problem in the launch
  int red_begin;       // first element of this problem in the partial-sum pass (upt > 1)
  long long part_off;  // first fp32 partial of this problem (used when upt > 1)
};
struct RowBatch {
  RowProb p[kMaxRankProblems];
  int n, units;
  int tile_rows;    // tokens per tile
  int unit_chunks;  // 64-wide reduction chunks per unit
  int red_total;    // elements of the partial-sum pass (0: none)
  float* partials;  // [tile][unit][tile_rows][rpad] per problem
  int* status;
  long long limit_ns;
};

// Column product problem: out_b[c, j] = sum_t X[t, c] * S_b[t, j] for every
// block b sharing X [T, C]; S_b is given transposed, S_b^T [rs_b, T]
// row-major.  out_cr: out_b[c * rs_b + j] (dB), else out_b[j * C + c] (dA).
struct ColProb {
  CUtensorMap tmX;                   // X [T, C]: box 64 columns x 64 tokens, 128-byte swizzle
  CUtensorMap tmS[kMaxRankBlocks];   // S_b^T [rs_b, T]: box 64 tokens x pad8(rs_b) rows, 128-byte swizzle
  int T, C;
  int nblk;
  int rs[kMaxRankBlocks];
  float* out[kMaxRankBlocks];
  int out_cr;
  int rpad;
  int tx_bytes;        // bytes of a full chunk stage (both X boxes + rank-side boxes)
  int upt;             // work units per 128-column tile (each unit_chunks x 64 tokens)
  int unit_begin;
  int red_begin;
  long long part_off;
};
struct ColBatch {
  ColProb p[kMaxRankProblems];
  int n, units;
  int tile_rows;    // columns per tile
  int unit_chunks;
  int red_total;
  float* partials;
  int* status;
  long long limit_ns;
};

// The backward's two products over dy in one pass (one problem per projection):
//   sv = s dy B   [T, r]   (bf16 into sv [T, ld_sv] and sv^T [pad8(r), T], zero columns / rows past r)
//   dB = dy^T su  [N, r]   (fp32)
// B and su come transposed (B^T [pad8(r), N], su^T [pad8(r), T], zero rows
// past r).  A work unit is (token group g, column piece q): the column blocks
// of q (128 columns each) in turn, and for each the group's 128-token tiles;
// the group's sv accumulators stay in TMEM across the unit.  A projection cut
// into several pieces writes fp32 sv partials [piece][T][rpad]; one cut into
// several groups writes fp32 dB partials [group][N][rpad]; the dy reduce pass
// sums them in order.
constexpr int kDyMaxCut = 8;  // most pieces / groups of one projection
struct DyProb {
  CUtensorMap tmDy;   // dy [T, N]: box 64 columns x 128 tokens, 128-byte swizzle
  CUtensorMap tmBt;   // B^T [r, N]: box 64 columns x pad8(r) rows
  CUtensorMap tmSuT;  // su^T [r, T]: box 64 tokens x pad8(r) rows
  int T, N, r, rpad;  // rpad: r rounded up to 16 (the MMA's N)
  float scale;
  __nv_bfloat16* sv;  // [T, ld_sv]
  int ld_sv;
  __nv_bfloat16* svT;  // [pad8(r), T]
  float* dB;           // [N, r]
  int tiles, tt, groups;     // 128-token tiles, tiles per group, groups
  int blocks, bpu, pieces;   // 128-column blocks, blocks per piece, pieces
  int unit_begin;
  long long sv_part, db_part;  // partial offsets (pieces > 1 / groups > 1)
};
struct DyBatch {
  DyProb p[kMaxRankProblems];
  int n, units;
  float* partials;
  int red_sv, red_db;  // items of the reduce pass: T x pad8(r) / 8 (pieces > 1), N x ceil(r / 4) (groups > 1)
  int* status;
  long long limit_ns;
};
// Largest token tiles per group for a padded rank (TMEM: sv accumulators of
// the group plus two dB accumulators).
int dy_tiles_max(int rpad);
cudaError_t launch_dy(const DyBatch& b, int ctas, cudaStream_t stream);

// Output rows (tokens of a row product, columns of a column product) per tile.
int rank_mma_tile();
// Rank-r products on the tensor cores, then their partial-sum pass when needed;
// `ctas` persistent CTAs (one per SM).
cudaError_t launch_rowmma(const RowBatch& b, int rmax, int ctas, cudaStream_t stream);
cudaError_t launch_colmma(const ColBatch& b, int rmax, int ctas, cudaStream_t stream);
cudaError_t launch_reduce_rows(const RowBatch& b, cudaStream_t stream);
cudaError_t launch_reduce_cols(const ColBatch& b, cudaStream_t stream);
// Batched transposes: dst_i[j, n] = src_i[n, j] for j < r_i, 0 for r_i <= j < r8_i
// (src_i [n_i, r_i] with row stride ld_i), every job in one launch.
constexpr int kMaxTransposes = 128;
struct TransposeJobs {
  const __nv_bfloat16* src[kMaxTransposes];
  __nv_bfloat16* dst[kMaxTransposes];
  int n[kMaxTransposes], r[kMaxTransposes], ld[kMaxTransposes], r8[kMaxTransposes];
  int count;
  long long max_elems;  // largest n_i * r8_i
};
cudaError_t launch_transposes(const TransposeJobs& jobs, cudaStream_t stream);

// ---------------------------------------------------------------- reduced-vocabulary cross entropy
// Index pass: J (ascending) = union of the trainable targets' first k top-k
// entries (every token when topk is null), pos[v] = column of v in J or -1,
// tl = trainable positions (ascending), tpos[t] = row of t in tl or -1,
// ycol[i] = column in J of the target of tl[i]; counts = {|tl|, |J|, bad
// input flag}.  flags (V bytes) and counts must be zero at launch.
struct CeIndex {
  const int32_t* targets;
  const uint8_t* mask;  // null: every position trainable
  int T, V;
  const int32_t* topk;  // [V, ld_topk], null: full vocabulary
  long long ld_topk;
  int k;
  uint8_t* flags;
  int32_t *J, *pos, *tl, *tpos, *ycol;
  int32_t* counts;      // [8]: |T_set|, |J|, error flag, -, two last-block counters
  int32_t* seg_counts;  // 128 per-segment counts of the vocabulary compaction
};
cudaError_t launch_ce_index(const CeIndex& a, cudaStream_t stream);
// dst[i, :] = src[idx[i], :] for i < n (rows of d bf16, d a multiple of 8).
cudaError_t launch_gather_rows(const __nv_bfloat16* src, long long ld, const int32_t* idx, int n, int d,
                               __nv_bfloat16* dst, cudaStream_t stream);
// Two such gathers in one launch.
cudaError_t launch_gather_rows2(const __nv_bfloat16* src_a, long long ld_a, const int32_t* idx_a, int n_a,
                                __nv_bfloat16* dst_a, const __nv_bfloat16* src_b, long long ld_b,
                                const int32_t* idx_b, int n_b, __nv_bfloat16* dst_b, int d, cudaStream_t stream);
// Per row i < nT of the fp32 logits Z [nT, ldz] with their log-sum-exp
// partials lse_part [nT, ld_part] (one per gemm_lse_group() columns), nT >= 1:
// lse[i], rowloss[i] = lse - z[ycol[i]] and G[i, :] = bf16(softmax - onehot),
// zero in columns [nJ, ldg).
// The last block also writes token_loss (optional) and *loss (as launch_ce_finish);
// done: a zeroed counter.
cudaError_t launch_ce_rows(const float2* lse_part, int ld_part, const float* Z, int ldz, int nJ, const int32_t* ycol,
                           int nT, float* lse, float* rowloss, const int32_t* tpos, int T, float* token_loss,
                           float* loss, int* done, __nv_bfloat16* G, int ldg, int num_sms, cudaStream_t stream);
// token_loss[t] (optional) and *loss = sum of rowloss in a fixed order.
cudaError_t launch_ce_finish(const float* rowloss, int nT, const int32_t* tpos, int T, float* token_loss,
                             float* loss, cudaStream_t stream);
// dst[t, :] = src[tpos[t], :] or zeros when tpos[t] < 0.
cudaError_t launch_scatter_rows(const __nv_bfloat16* src, const int32_t* tpos, int T, int d, __nv_bfloat16* dst,
                                cudaStream_t stream);

// ---------------------------------------------------------------- top-k similarity table
// En[i] = bf16(E[i] / ||E[i]||), the norm's sum of squares in fp32 in index order.
cudaError_t launch_normalize_rows(const __nv_bfloat16* E, int V, int d, __nv_bfloat16* En, cudaStream_t stream);
// Rows row0 .. row0 + nrows - 1 of the table from their similarities S [nrows, lds] fp32:
// the k largest per row, descending, lower index first on ties; *status =
// kStatusTopkTies when a row has too many candidates tied at its k-th value.
// Top-k selection per row of similarities S [nrows, lds] (row r goes to table
// row rows[r], or row0 + r when rows is null).
cudaError_t launch_topk_select(const float* S, long long lds, int V, int k, int row0, const int32_t* rows, int nrows,
                               int32_t* table, int* status, cudaStream_t stream);
// Thresholds of nrows rows from their sample similarities Z [nrows, topk_sample()].
cudaError_t launch_topk_tau(const float* Z, int V, int k, int nrows, float* tau, cudaStream_t stream);
// Sorts each row's appended candidates into the table (a warp per row, a block for
// lists over 1024: big_rows / big_count, a zeroed count), or lists the row for the fallback.
cudaError_t launch_topk_sort(const uint2* cand, int* cnt, int cap, int k, int row0, int nrows, int32_t* table,
                             int32_t* big_rows, int* big_count, int32_t* fail_rows, int* fail_count, int num_sms,
                             cudaStream_t stream);
// Es [topk_sample(), d] = the evenly spread sample rows of En [V, d].
cudaError_t launch_topk_gather_sample(const __nv_bfloat16* En, int V, int d, __nv_bfloat16* Es, int num_sms,
                                      cudaStream_t stream);
int topk_sample();        // sample tokens per row
int topk_sample_min_v();  // shortest rows that take the sampled selection
int topk_cap();           // candidate slots per row
int topk_max_k();

// One bounded wait on a barrier nothing arrives on (failure-detection self-check).
cudaError_t launch_wait_probe(int* status, long long limit_ns, cudaStream_t stream);

// dst[i, j] = j < r ? src[i * r + j] : 0  for j < ld_dst (zero-padded copy of an [rows, r] matrix).
cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t stream);

}  // namespace lora
