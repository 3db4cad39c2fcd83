/*
 * lora.h -- C ABI of the GB300 (sm_103a) LoRA-adapted linear layer.
 *
 * The operation.  A frozen linear layer W is adapted by a trainable rank-r
 * product, as in the LoRA fine-tuning the paper studies (Background,
 * "Parameter-Efficient Fine-Tuning": low-rank decomposition matrices trained
 * while the original weights stay frozen; rank r and alpha from the
 * hyper-parameter table; s = alpha / r).  Token-major, row-major layout:
 *
 *   forward   su = s * x A^T                [T, r]   (saved for backward)
 *             y  = x W^T + su B^T           [T, N]
 *   backward  sv = s * dy B                 [T, r]   (internal)
 *             dx = dy W + sv A              [T, K]
 *             dB = dy^T su                  [N, r]   (= s dy^T x A^T)
 *             dA = sv^T x                   [r, K]   (= s (dy B)^T x)
 *
 * y = x W^T and dx = dy W are Algorithm 1's y_base = W x and dx = W^T dy
 * (column-vector form there).  W is frozen: no gradient of W is formed.
 *
 * Shapes: T tokens, K = d_in, N = d_out, r = rank.  x [T,K], W [N,K]
 * (nn.Linear layout), A [r,K], B [N,r], y and dy [T,N], dx [T,K], su [T,r].
 * Element types: every activation and parameter is bf16 (passed as its
 * 16-bit pattern, `lora_bf16`); contractions accumulate in fp32; y, dx and su
 * are rounded to bf16 (round to nearest even) once; dA and dB are fp32.
 *
 * Conventions shared by every entry point:
 *  - every pointer is a CUDA device pointer on the current device, owned by
 *    the caller, row-major and dense (leading dimension = row length), and
 *    16-byte aligned; the library never allocates or frees memory;
 *  - T, d_in and d_out are multiples of 8 (16-byte rows for the tensor-memory
 *    accelerator), 0 <= rank <= 128, scale finite;
 *  - rank 0 is a frozen projection without an adapter: the forward computes
 *    y = x W^T and the backward dx = dy W only; A, B, su, dA and dB are
 *    neither read nor written and may be NULL.  The paper adapts only the q
 *    and v projections of each layer (hyper-parameter table), so the other
 *    projections of a layer are such frozen linears, still on the backward
 *    path through dx;
 *  - calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *    default stream); return LORA_OK once every kernel is enqueued;
 *  - inputs may alias each other (e.g. q, k and v passing one x); outputs
 *    must not alias any input or each other; W is never written;
 *  - dA and dB are overwritten, not accumulated;
 *  - `workspace` is scratch of at least the size the matching
 *    *_workspace_size call reports, 256-byte aligned; its contents need no
 *    initialisation and are garbage afterwards; calls that run concurrently
 *    need separate workspaces;
 *  - errors: a negative LORA_E* code is returned and nothing is enqueued
 *    (argument errors), or kernels may already be enqueued (LORA_ECUDA);
 *    lora_last_error() repeats the code the calling thread's latest call
 *    returned.
 *    Device-side bounded waits that expire set a status word readable with
 *    lora_read_status (LORA_ETIMEOUT); they never trap.
 *
 * Environment (read once per process; for measurement, never needed):
 *   LORA_PDL=0        launch without programmatic dependent launch;
 *   LORA_OVERLAP=0    run a forward-and-backward call on the caller's stream
 *                     alone (no side stream for the backward's rank-r work);
 *   LORA_SIDE_SMS=n   SMs of the side stream beside the forward contraction,
 *   LORA_SIDE_SMS2=n  and beside the backward-dx contraction (2 .. SMs / 4;
 *                     default: the balance rule of the implementation).
 * A workspace size reported with one setting may not cover a call made with
 * another: query the size in the process that makes the calls.
 */
#ifndef LORA_GB300_H_
#define LORA_GB300_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t lora_bf16; /* bit pattern of an IEEE bfloat16 */

enum {
  LORA_OK = 0,
  LORA_EINVAL = -1,      /* bad shape, rank, scale, mode or count */
  LORA_ENULL = -2,       /* a required pointer is NULL */
  LORA_EALIGN = -3,      /* a pointer is not 16-byte aligned (workspace: 256) */
  LORA_ECUDA = -4,       /* a CUDA runtime call or launch failed */
  LORA_ETIMEOUT = -5,    /* a device-side bounded wait expired */
  LORA_EWORKSPACE = -6,  /* workspace missing or smaller than required */
  LORA_EDEVICE = -7,     /* current device is not a compute capability 10.3 GPU */
  LORA_ESCRATCH = -8     /* needs more scratch than lora_linear_fwd_noalloc's fixed array */
};

enum { LORA_FWD = 1, LORA_BWD = 2, LORA_FWD_BWD = 3 };

typedef struct lora_shape {
  int64_t T;      /* tokens */
  int64_t d_in;   /* K */
  int64_t d_out;  /* N */
  int64_t rank;   /* r */
  float scale;    /* s = alpha / r */
} lora_shape;

/* Bytes of workspace that lora_linear_fwd (mode LORA_FWD), lora_linear_bwd
 * (LORA_BWD) or both (LORA_FWD_BWD) need for `shape`.
 * Returns LORA_OK, LORA_EINVAL or LORA_ENULL. */
int lora_workspace_size(const lora_shape* shape, int mode, size_t* bytes);

/* Forward of one LoRA linear: y = x W^T + s (x A^T) B^T.
 * su [T,r] receives s x A^T for the backward; pass NULL for a forward that
 * saves nothing (the no-grad forward of a checkpointed schedule).
 * Reads x, W, A, B; writes y and su. */
int lora_linear_fwd(const lora_shape* shape, const lora_bf16* x, const lora_bf16* W,
                    const lora_bf16* A, const lora_bf16* B, lora_bf16* y, lora_bf16* su,
                    void* workspace, size_t workspace_bytes, void* stream);

/* Forward of one LoRA linear as lora_linear_fwd computes it, but with no
 * workspace argument, for callers that cannot allocate device memory when
 * they call: an operator running inside another framework's execution
 * callback, where allocating is not allowed, or a latency-bound path that
 * cannot afford the device-wide synchronisation cudaMalloc and cudaFree
 * cause.  Its scratch is one fixed array of 4 MiB in device memory that the
 * library owns; every GPU that loads the library keeps it until the process
 * exits.  Shapes whose forward needs more scratch than that are rejected
 * with LORA_ESCRATCH before anything is enqueued (roughly when tokens x
 * d_in x rank reaches 2^29; 4096 tokens x d_in 4096 at rank 16 fit).  The
 * first call on a device looks up the array's device address; make that
 * first call before any stream capture.
 * All calls share the array and leave their scratch in it: calls that
 * overlap on the GPU (for example on two streams at once) race and give
 * wrong results.  Nothing is allocated.  It never stores fp32 partial sums
 * of a contraction: lora_linear_fwd may cut the contraction of a forward
 * with few output tiles (fewer than 76 of 256 x 512) into fp32 partials in
 * its workspace when the two CTA pairs of a cluster cannot share it, and
 * there the two results differ by the bf16 rounding of differently ordered
 * fp32 sums; everywhere else (76 or more tiles, or a contraction shared
 * within clusters, as for 512 tokens x d_out 3072) they are identical bit
 * for bit.  The paper has no counterpart of this entry point.  Returns as
 * lora_linear_fwd (argument errors first), or LORA_ESCRATCH. */
int lora_linear_fwd_noalloc(const lora_shape* shape, const lora_bf16* x, const lora_bf16* W,
                            const lora_bf16* A, const lora_bf16* B, lora_bf16* y, lora_bf16* su,
                            void* stream);

/* Backward of one LoRA linear with W frozen.
 * su is the forward's saved s x A^T.  dx may be NULL (no input gradient
 * wanted); dA [r,K] and dB [N,r] are required.  Reads dy, x, W, A, B, su. */
int lora_linear_bwd(const lora_shape* shape, const lora_bf16* dy, const lora_bf16* x,
                    const lora_bf16* W, const lora_bf16* A, const lora_bf16* B,
                    const lora_bf16* su, lora_bf16* dx, float* dA, float* dB,
                    void* workspace, size_t workspace_bytes, void* stream);

/* Frozen base weight in 4-bit form, dequantized on the fly inside the fused
 * contractions (Algorithm 1, "On-the-fly Dequantization": W = s * W_q + b,
 * rematerialized for the forward and again for the backward, never kept):
 * the bf16 W is never written to memory.  One (s, b) pair per output row n
 * and group of 64 consecutive input columns k = 64 g .. 64 g + 63; each
 * dequantized element is bf16(s * q + b), rounded once.  The paper fixes
 * neither the group size nor the code layout; these are the library's:
 *   codes   [d_out][d_in / 2] bytes, codes q[n][k] in 0..15.  The
 *           little-endian 32-bit word m of row n covers k = 8m .. 8m + 7:
 *           q[n][8m + 2i] in bits 4i .. 4i + 3 and q[n][8m + 2i + 1] in bits
 *           16 + 4i .. 16 + 4i + 3, for i = 0..3;
 *   params  [d_out][d_in / 64][2] bf16: (s, b) of row n, group g.
 * d_in must be a multiple of 256; both pointers 16-byte aligned. */
typedef struct lora_q4_weight {
  const uint8_t* codes;
  const lora_bf16* params;
} lora_q4_weight;

/* As lora_linear_fwd / lora_linear_bwd with the base weight given as 4-bit
 * codes (lora_q4_weight) instead of bf16 W.  Returns LORA_EINVAL when d_in is
 * not a multiple of 256. */
int lora_linear_fwd_q4(const lora_shape* shape, const lora_bf16* x, const lora_q4_weight* Wq,
                       const lora_bf16* A, const lora_bf16* B, lora_bf16* y, lora_bf16* su,
                       void* workspace, size_t workspace_bytes, void* stream);
int lora_linear_bwd_q4(const lora_shape* shape, const lora_bf16* dy, const lora_bf16* x,
                       const lora_q4_weight* Wq, const lora_bf16* A, const lora_bf16* B,
                       const lora_bf16* su, lora_bf16* dx, float* dA, float* dB,
                       void* workspace, size_t workspace_bytes, void* stream);

/* One adapted projection of a decoder layer (q, k, v, o, gate, up, down).
 * Field meanings and rules as above; pointers a mode does not touch may be
 * NULL (forward: x W A B y [su]; backward: dy x W A B su dA dB [dx]).  The
 * base weight is either W (bf16) or Wq (4-bit; then W must be NULL). */
typedef struct lora_proj {
  lora_shape shape;
  const lora_bf16* x;
  const lora_bf16* W;
  const lora_bf16* A;
  const lora_bf16* B;
  const lora_bf16* dy;
  lora_bf16* y;
  lora_bf16* su;
  lora_bf16* dx;
  float* dA;
  float* dB;
  lora_q4_weight Wq;
} lora_proj;

/* Workspace bytes for lora_stack_step over `projs` in `mode`. */
int lora_stack_workspace_size(const lora_proj* projs, int n_proj, int mode, size_t* bytes);

/* Forward and/or backward of n_proj independent projections (1..64), e.g.
 * the seven adapted linears of one decoder layer.  Mode LORA_FWD_BWD runs
 * every forward, then every backward.  Same semantics as n_proj calls of
 * lora_linear_fwd / lora_linear_bwd, scheduled as one batch on `stream`. */
int lora_stack_step(const lora_proj* projs, int n_proj, int mode, void* workspace,
                    size_t workspace_bytes, void* stream);

/* Memory-efficient checkpointed schedule over a stack of layers
 * (Algorithm 2, "forward twice, backward once"): Stage I runs the forward of
 * every layer without saving anything (as with su = NULL); Stage III walks
 * the layers from the last to the first and for each re-runs its forward,
 * keeping su only in the workspace, then its backward.  Only the layers'
 * inputs (x, and dy for the backward) need to stay resident between the
 * stages; no su of any layer outlives its backward.  `projs` holds
 * n_layers x n_per_layer projections, layer-major, each with x, W (or Wq),
 * A, B, dy, y, dA, dB (dx optional); their su fields are ignored.  y is
 * written by both stages (with the same values).  Results equal those of
 * lora_stack_step(LORA_FWD_BWD) layer by layer.  n_per_layer 1..64.
 * Returns as lora_stack_step. */
int lora_stack_ckpt_workspace_size(const lora_proj* projs, int n_layers, int n_per_layer, size_t* bytes);
int lora_stack_ckpt(const lora_proj* projs, int n_layers, int n_per_layer, void* workspace,
                    size_t workspace_bytes, void* stream);

/* Reduced-vocabulary LM-head cross entropy with logits masking (Sections
 * "Softmax Approximation" and "Logits Masking").  Hidden states h [T, d]
 * enter the frozen LM head E [V, d] (one row per vocabulary token).  With
 * trainable positions T_set (mask) and targets y, the reduced vocabulary is
 *     J = union over t in T_set of topk[y_t, 0..k-1]     (every token when topk is NULL)
 * logits are formed only for t in T_set and only over J:
 *     z_t[j] = h_t . E_j,   loss = sum_{t in T_set} (log sum_{j in J} exp z_t[j] - z_t[y_t])
 * and the only gradient (E frozen) is
 *     dh_t = sum_{j in J} (softmax_J(z_t)[j] - [j == y_t]) E_j for t in T_set, 0 elsewhere.
 * Row i of the top-k table lists tokens by descending similarity to token i
 * and starts with i (so every trainable target is in J); it is the table
 * lora_topk_table builds.  The call synchronizes `stream` once, after the
 * index pass, to size the two contractions by |T_set| and |J| (so it cannot
 * be captured into a CUDA graph).  Logits are accumulated in fp32 and kept in
 * fp32; softmax - onehot enters the dh contraction in bf16; dh is bf16.
 * Requirements: d a multiple of 8, T >= 1, V >= 1, 1 <= k <= ld_topk; targets
 * of trainable positions in [0, V) and table entries in [0, V) (else
 * LORA_EINVAL after the index pass, outputs untouched). */
typedef struct lora_ce_args {
  int64_t T, d, V;
  const lora_bf16* h;       /* [T, d] */
  const lora_bf16* E;       /* [V, d] */
  const int32_t* targets;   /* [T] */
  const uint8_t* mask;      /* [T], nonzero = trainable; NULL = every position */
  const int32_t* topk;      /* [V, ld_topk], or NULL for the full vocabulary */
  int64_t ld_topk, k;
  float* loss;              /* [1]: the sum over trainable positions */
  float* token_loss;        /* [T] or NULL: per-position losses, 0 off T_set */
  lora_bf16* dh;            /* [T, d] or NULL (no backward) */
  int32_t* vocab;           /* [V] or NULL: receives J in ascending order */
  int64_t* counts;          /* host [2] or NULL: receives |T_set| and |J| */
} lora_ce_args;

/* Workspace bytes for the worst case |T_set| = T, |J| = V. */
int lora_ce_workspace_size(const lora_ce_args* args, size_t* bytes);
int lora_ce_fwd_bwd(const lora_ce_args* args, void* workspace, size_t workspace_bytes, void* stream);

/* Top-k similarity table of a frozen embedding (Section "Softmax
 * Approximation", "Choosing the Reduced Vocabulary Set"): with E~ the
 * embedding's rows normalised (each row's sum of squares accumulated in fp32
 * in index order, correctly rounded square root and division, rounded to
 * bf16; a zero row stays zero), C = E~ E~^T holds the cosine similarities and
 * row i of `table` [V, k] int32 lists the k tokens with the largest C[i, :],
 * in descending order, the lower index first on equal similarities (row i
 * starts with i unless another token has the same direction).  The V x V
 * matrix is never formed.  Below V = 32768 similarities are computed 512 rows
 * at a time in fp32 on the tensor cores and each row's top k is selected from
 * them.  From V = 32768 on, each row first gets a threshold from its
 * similarities to 8192 evenly spread tokens, the similarity contraction keeps
 * only the values at or above it (at most 4096 per row, in workspace), and
 * those are sorted; rows left with fewer than k or more than 4096 such values
 * are redone exactly on the 512-row path, which needs one synchronization of
 * `stream` (a 4-byte read of their count) before the call returns.
 * E [V, d] bf16 (16-byte aligned), d a multiple of 8, 1 <= k <= min(V, 1024).
 * A row whose k-th similarity is shared by more candidates than the selection
 * holds (thousands of exact ties) is left unwritten and lora_read_status
 * reports LORA_EINVAL. */
int lora_topk_workspace_size(int64_t V, int64_t d, int64_t k, size_t* bytes);
int lora_topk_table(const lora_bf16* E, int64_t V, int64_t d, int64_t k, int32_t* table, void* workspace,
                    size_t workspace_bytes, void* stream);

/* Waits for `stream`, then reads the device status word that bounded waits
 * set when they expire (and lora_topk_table sets on an unresolved row):
 * *status = LORA_OK, LORA_ETIMEOUT or LORA_EINVAL.  reset != 0 clears it.
 * Returns LORA_OK or LORA_ECUDA. */
int lora_read_status(void* stream, int* status, int reset);

/* Failure-detection self-check (the paper has no counterpart): enqueues one
 * kernel that waits, with the same bounded wait every kernel of the library
 * uses, on a barrier nothing arrives on.  After limit_ns (1 us .. 1 s) of
 * device time the wait gives up, records LORA_ETIMEOUT in the status word and
 * the kernel returns, leaving the context usable; lora_read_status then
 * reports LORA_ETIMEOUT.  Returns LORA_OK once enqueued, LORA_EINVAL for a
 * limit out of range. */
int lora_wait_selftest(int64_t limit_ns, void* stream);

/* Limit, in nanoseconds of device time, of every bounded wait in the
 * library's kernels (0 restores the default of 4 s).  For tests of the
 * timeout path; affects launches made after the call.  Returns LORA_OK. */
int lora_set_wait_limit_ns(int64_t ns);

/* Kernel kinds of the profiling interface below. */
enum {
  LORA_KERNEL_GEMM_FWD = 0, /* fused [x | su] . [W | B]^T contraction */
  LORA_KERNEL_GEMM_BWD = 1, /* fused [dy | sv] . [W ; A] contraction */
  LORA_KERNEL_ROWPROJ = 2,  /* su = s x A^T; the pass over dy: sv = s dy B, and dB = dy^T su where fused
                               (r <= 16); with their partial sums */
  LORA_KERNEL_COLPROJ = 3,  /* dA = sv^T x, and dB = dy^T su where not fused; with their partial sums */
  LORA_KERNEL_PAD = 4,      /* zero-padded copies for ranks that are not multiples of 8 */
  LORA_KERNEL_KINDS = 5
};

/* Number of kernels the library has enqueued since it was loaded (all
 * devices).  A call rejected with an argument error enqueues none. */
int64_t lora_launch_count(void);

/* Device-time profiling: after lora_profile_begin, every launch group of
 * the library is bracketed by CUDA events recorded on its stream.
 * lora_profile_end waits for those events, writes the summed device time in
 * milliseconds and the kernel launches per kind into ms[LORA_KERNEL_KINDS]
 * and launches[LORA_KERNEL_KINDS] (either may be NULL), and stops recording.
 * Returns LORA_OK, LORA_EINVAL (end without begin) or LORA_ECUDA. */
int lora_profile_begin(void);
/* As lora_profile_begin, but only the launch groups of the kinds whose bit
 * (1u << LORA_KERNEL_*) is set in kind_mask are bracketed; the others run
 * with no event between their launches. */
int lora_profile_begin_kinds(uint32_t kind_mask);
int lora_profile_end(double* ms, int64_t* launches);

/* Static message for a LORA_* code. */
const char* lora_strerror(int code);

/* The code the calling thread's most recent library call returned (every
 * entry point that returns a LORA_* code records it, successes included, in
 * thread-local storage; lora_strerror, lora_version, lora_launch_count and
 * lora_last_error itself do not).  Device-side codes of kernels that already
 * ran are not included: lora_read_status reports those.  LORA_OK before any
 * call.  For callers that keep only a success flag across a layer of their
 * own; each call also returns its code directly. */
int lora_last_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int lora_version(void);

#ifdef __cplusplus
}
#endif

#endif /* LORA_GB300_H_ */
