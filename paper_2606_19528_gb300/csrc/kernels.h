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
  int num_m_tiles;
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
  CUtensorMap tmOut[kMaxProblems];  // out [M, N]: 64 columns x 32 rows boxes, 128-byte swizzle
  GemmProblem prob[kMaxProblems];
  int num_problems;
  int total_tiles;
  int* tile_counter;   // zero at launch; hands out tiles in list order
  int* status;
  long long limit_ns;
};

cudaError_t launch_fused_gemm(const GemmBatch& batch, bool b_mn_major, int num_sms, cudaStream_t stream);
size_t fused_gemm_smem_bytes();
int gemm_tile_m();
int gemm_tile_n();
int gemm_tile_k();

// ---------------------------------------------------------------- rank-r kernels
inline int rank_pad16(int r) { return (r + 15) / 16 * 16; }
inline int rank_pad8(int r) { return (r + 7) / 8 * 8; }

constexpr int kMaxRankBlocks = 4;     // projections fused into one problem
constexpr int kMaxRankProblems = 12;  // problems per launch

// Row product problem: out_b[t, j] = scale * sum_c X[t, c] * Wv_b(j, c) for
// every block b (one projection each) sharing the activation X [T, C].
//   w_rc launches: Wv_b(j, c) = W_b[j * ldw_b + c]   (A of the adapter, [r_b, C])
//   otherwise:     Wv_0(j, c) = W_0[c * ldw_0 + j]   (B of the adapter, [C, r]; one block)
// Blocks are concatenated at 8-aligned rank offsets; columns rw_b .. ld_out_b
// of out_b are written as zeros; out2_b (optional) gets columns < ld_out2_b.
struct RowProb {
  CUtensorMap tmX;                   // X [T, C]: box 64 columns x 64 tokens, 128-byte swizzle
  CUtensorMap tmW[kMaxRankBlocks];   // w_rc: A_b [r_b, C], box 64 x pad8(r_b), 128-byte swizzle;
                                     // else: B [C, r] (one block), box pad8(r) x 64, no swizzle
  int T, C;
  int nblk;
  int rw[kMaxRankBlocks];
  __nv_bfloat16* out[kMaxRankBlocks];
  int ld_out[kMaxRankBlocks];
  __nv_bfloat16* out2[kMaxRankBlocks];
  int ld_out2[kMaxRankBlocks];
  float scale;
  int rpad;            // concatenated rank, rounded up to 16
  int tx_bytes;        // bytes one chunk stage receives (X box + rank-side boxes)
  int upt;             // work units per 64-token tile (each unit_chunks x 64 columns)
  int unit_begin;      // first unit of this problem in the launch
  int red_begin;       // first element of this problem in the reduction pass (upt > 1)
  long long part_off;  // first fp32 partial of this problem (used when upt > 1)
};
struct RowBatch {
  RowProb p[kMaxRankProblems];
  int n, units, w_rc;
  int unit_chunks;  // 64-wide reduction chunks per unit
  int red_total;    // elements of the reduction pass (0: none)
  float* partials;  // [tile][unit][64][rpad] per problem
  int* status;
  long long limit_ns;
};

// Column product problem: out_b[c, j] = sum_t X[t, c] * S_b[t, j] for every
// block b sharing X [T, C]; S_b is [T, pad8(rs_b)] with zeros beyond rs_b.
// out_cr: out_b[c * rs_b + j] (dB), else out_b[j * C + c] (dA).
struct ColProb {
  CUtensorMap tmX;                   // X [T, C]: box 64 columns x 64 tokens, 128-byte swizzle
  CUtensorMap tmS[kMaxRankBlocks];   // S_b: box pad8(rs_b) x 64 tokens, no swizzle
  int T, C;
  int nblk;
  int rs[kMaxRankBlocks];
  float* out[kMaxRankBlocks];
  int out_cr;
  int rpad;
  int tx_bytes;
  int upt;             // work units per 64-column tile (each unit_chunks x 64 tokens)
  int unit_begin;
  int red_begin;
  long long part_off;
};
struct ColBatch {
  ColProb p[kMaxRankProblems];
  int n, units;
  int unit_chunks;
  int red_total;
  float* partials;
  int* status;
  long long limit_ns;
};

int rank_tile();
cudaError_t launch_rowprod(const RowBatch& b, int rmax, int num_sms, cudaStream_t stream);
cudaError_t launch_colprod(const ColBatch& b, int rmax, int num_sms, cudaStream_t stream);

// dst[i, j] = j < r ? src[i * r + j] : 0  for j < ld_dst (zero-padded copy of an [rows, r] matrix).
cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t stream);

}  // namespace lora
