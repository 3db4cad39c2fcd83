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
  int* status;
  long long limit_ns;
};

cudaError_t launch_fused_gemm(const GemmBatch& batch, bool b_mn_major, int num_sms, cudaStream_t stream);
size_t fused_gemm_smem_bytes();
int gemm_tile_m();
int gemm_tile_n();
int gemm_tile_k();

// ---------------------------------------------------------------- rank-r kernels
// Padded rank used by the rank-r kernels: r rounded up to a multiple of 16.
inline int rank_pad16(int r) { return (r + 15) / 16 * 16; }
inline int rank_pad8(int r) { return (r + 7) / 8 * 8; }

// Row products  out[t, j] = scale * sum_c X[t, c] * Wv(j, c),  t < T, j < r.
//   w_rc = true : Wv(j, c) = Wm[j * ldw + c]   (A of the adapter, [r, C])
//   w_rc = false: Wv(j, c) = Wm[c * ldw + j]   (B of the adapter, [C, r]; ldw % 8 == 0)
// The reduction over c is split across `splits` CTA columns; with splits > 1
// fp32 partials go to `part` [splits, T, r] and reduce_rows finishes.
struct RowProjPlan {
  int splits;
  int chunks_per_split;  // 64-wide column chunks per split
};
RowProjPlan plan_rowproj(int T, int C, int num_sms);
cudaError_t launch_rowproj(const __nv_bfloat16* X, int ldx, const __nv_bfloat16* Wm, int ldw, bool w_rc,
                           int T, int C, int r, const RowProjPlan& plan, float* part,
                           __nv_bfloat16* out, int ld_out, __nv_bfloat16* out2, int ld_out2, float scale,
                           cudaStream_t stream);

// Column products  G[c, j] = sum_t X[t, c] * S[t, j],  c < C, j < r  (S: lds % 8 == 0).
//   out_cr = true : out[c * r + j]   ([C, r], dB)
//   out_cr = false: out[j * C + c]   ([r, C], dA)
struct ColProjPlan {
  int splits;
  int chunks_per_split;  // 64-token chunks per split
};
ColProjPlan plan_colproj(int T, int C, int num_sms);
cudaError_t launch_colproj(const __nv_bfloat16* X, int ldx, const __nv_bfloat16* S, int lds, int T, int C,
                           int r, const ColProjPlan& plan, float* part, float* out, bool out_cr,
                           cudaStream_t stream);

// dst[i, j] = j < r ? src[i * r + j] : 0  for j < ld_dst (zero-padded copy of an [rows, r] matrix).
cudaError_t launch_pad_cols(const __nv_bfloat16* src, int rows, int r, __nv_bfloat16* dst, int ld_dst,
                            cudaStream_t stream);

}  // namespace lora
