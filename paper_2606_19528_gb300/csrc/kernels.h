// Internal interface between the C ABI (api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace lora {

// Counts one kernel launch (defined with the C ABI).
void note_launch();

// ---------------------------------------------------------------- fused GEMM
constexpr int kMaxProblems = 8;

struct GemmProblem {
  __nv_bfloat16* out;  // [M, N] bf16, leading dimension ldo
  int ldo;
  int M;               // tokens
  int N;               // output columns
  int Kmain;           // base contraction length
  int r;               // adapter slab length (rank)
  int num_n_tiles;     // tiles along N
  int tile_begin;      // first index of this problem in the batch's tile list
  int kb_main;         // contraction blocks of the base part
  int kb_total;        // base + adapter blocks
  int m_fast;          // 1: consecutive tiles walk M (the weight tile stays put)
  int num_m_tiles;     // super-tiles (pairs x 256 rows) along M
};

// One launch: up to kMaxProblems independent fused contractions.
//  tmA  [M, Kmain] K-major (x or dy)        tmA2 [M, r] K-major (su or sv)
//  forward:  tmB  W [N, Kmain] K-major       tmB2 B [N, r] K-major
//  backward: tmB  W [Kmain, N] MN-major      tmB2 A [r, N] MN-major
struct GemmBatch {
  CUtensorMap tmA[kMaxProblems];
  CUtensorMap tmA2[kMaxProblems];
  CUtensorMap tmB[kMaxProblems];
  CUtensorMap tmB2[kMaxProblems];
  GemmProblem prob[kMaxProblems];
  int num_problems;
  int total_tiles;
  int* tile_counter;   // zero at launch; hands out tiles in list order
  int* status;
  long long limit_ns;
};

// pairs: CTA pairs per cluster (1, or 2 to share the weight tile between two
// vertically adjacent tiles); tiles of the batch must have been counted for it.
cudaError_t launch_fused_gemm(const GemmBatch& batch, bool b_mn_major, int pairs, int num_sms, cudaStream_t stream);
size_t fused_gemm_smem_bytes();
int gemm_tile_m();
int gemm_tile_n();
int gemm_tile_k();

// ---------------------------------------------------------------- rank-r kernels
inline int rank_pad16(int r) { return (r + 15) / 16 * 16; }
inline int rank_pad8(int r) { return (r + 7) / 8 * 8; }

constexpr int kMaxRankBlocks = 4;     // projections fused into one problem
constexpr int kMaxRankProblems = 16;  // problems per launch

// Row product problem: out_b[t, j] = scale * sum_c X[t, c] * Wv_b(j, c) for
// every block b (one projection each) sharing the activation X [T, C].
//   w_rc launches: Wv_b(j, c) = W_b[j * ldw_b + c]   (A of the adapter, [r_b, C])
//   otherwise:     Wv_0(j, c) = W_0[c * ldw_0 + j]   (B of the adapter, [C, r]; one block)
// Blocks are concatenated at 8-aligned rank offsets; columns rw_b .. ld_out_b
// of out_b are written as zeros; out2_b (optional) gets columns < ld_out2_b.
struct RowProb {
  const __nv_bfloat16* X;
  int ldx, T, C;
  int nblk;
  const __nv_bfloat16* W[kMaxRankBlocks];
  int ldw[kMaxRankBlocks];
  int rw[kMaxRankBlocks];
  __nv_bfloat16* out[kMaxRankBlocks];
  int ld_out[kMaxRankBlocks];
  __nv_bfloat16* out2[kMaxRankBlocks];
  int ld_out2[kMaxRankBlocks];
  float scale;
  int rpad;        // concatenated rank, rounded up to 16
  int cps;         // 64-column chunks per split
  int tile_begin;  // first 64-token tile of this problem in the launch
};
struct RowBatch {
  RowProb p[kMaxRankProblems];
  int n, tiles, splits, w_rc;
};

// Column product problem: out_b[c, j] = sum_t X[t, c] * S_b[t, j] for every
// block b sharing X [T, C]; S_b has row stride lds_b (a multiple of 8) and
// zeros in columns rs_b .. pad8(rs_b).  out_cr: out_b[c * rs_b + j] (dB),
// else out_b[j * C + c] (dA).
struct ColProb {
  const __nv_bfloat16* X;
  int ldx, T, C;
  int nblk;
  const __nv_bfloat16* S[kMaxRankBlocks];
  int lds[kMaxRankBlocks];
  int rs[kMaxRankBlocks];
  float* out[kMaxRankBlocks];
  int out_cr;
  int rpad;
  int cps;         // 64-token chunks per split
  int tile_begin;  // first 64-column tile of this problem in the launch
};
struct ColBatch {
  ColProb p[kMaxRankProblems];
  int n, tiles, splits;
};

int rank_tile();
// Cluster size (1, 2, 4 or 8) splitting each reduction so that the launch fills the GPU.
int rank_splits(int tiles, int max_chunks, int num_sms);
cudaError_t launch_rowprod(const RowBatch& b, int rmax, cudaStream_t stream);
cudaError_t launch_colprod(const ColBatch& b, int rmax, cudaStream_t stream);

// dst[i, j] = j < r ? src[i * r + j] : 0  for j < ld_dst (zero-padded copy of an [rows, r] matrix).
cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t stream);

}  // namespace lora
