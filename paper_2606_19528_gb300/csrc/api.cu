// C ABI of the LoRA linear (declared in include/lora.h): argument checks,
// workspace planning, TMA descriptors and the launch sequence.
//
// forward  : su = s x A^T (row product)  ->  y = [x | su] . [W | B]^T (fused GEMM)
// backward : sv = s dy B (row product), dB = dy^T su, dA = sv^T x (column
//            products)  ->  dx = [dy | sv] . [W ; A] (fused GEMM)
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>
#include <vector>

#include "common.cuh"
#include "kernels.h"
#include "lora.h"

namespace lora {
namespace {

__device__ int g_status;  // first device-side error (kStatusTimeout), 0 if none

constexpr int kMaxDevices = 64;
constexpr size_t kWsHeader = 256;  // 64 tile counters, one per fused-GEMM launch of a call
constexpr long long kDefaultWaitNs = 4000000000ll;

struct DeviceInfo {
  bool ready = false;
  bool supported = false;
  int num_sms = 0;
  int* status = nullptr;
};

std::mutex g_mu;
DeviceInfo g_dev[kMaxDevices];
long long g_wait_limit_ns = kDefaultWaitNs;

// ------------------------------------------------------------------ launch count and profiling
std::atomic<long long> g_launches{0};

struct ProfRec {
  int kind;
  cudaEvent_t a, b;
  long long launches;
};

struct Profiler {
  bool on = false;
  std::vector<cudaEvent_t> pool;  // events are reused across sessions
  size_t next = 0;
  std::vector<ProfRec> recs;
  cudaEvent_t take() {
    if (next == pool.size()) {
      cudaEvent_t e = nullptr;
      if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
      pool.push_back(e);
    }
    return pool[next++];
  }
};

std::mutex g_prof_mu;
Profiler g_prof;

// Brackets one launch group with CUDA events while a profiling session is on.
class ProfScope {
 public:
  ProfScope(int kind, cudaStream_t st) : kind_(kind), st_(st) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof.on) return;
    a_ = g_prof.take();
    b_ = g_prof.take();
    if (a_ && b_ && cudaEventRecord(a_, st_) == cudaSuccess) {
      active_ = true;
      l0_ = g_launches.load();
    }
  }
  ~ProfScope() {
    if (!active_) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (g_prof.on && cudaEventRecord(b_, st_) == cudaSuccess)
      g_prof.recs.push_back(ProfRec{kind_, a_, b_, g_launches.load() - l0_});
  }

 private:
  int kind_;
  cudaStream_t st_;
  cudaEvent_t a_ = nullptr, b_ = nullptr;
  bool active_ = false;
  long long l0_ = 0;
};

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn g_encode = nullptr;

int device_info(DeviceInfo** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LORA_ECUDA;
  std::lock_guard<std::mutex> lk(g_mu);
  DeviceInfo& d = g_dev[dev];
  if (!d.ready) {
    int major = 0, minor = 0, sms = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return LORA_ECUDA;
    d.supported = (major == 10 && minor == 3);
    d.num_sms = sms;
    if (d.supported) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_status) != cudaSuccess) return LORA_ECUDA;
      d.status = static_cast<int*>(p);
    }
    if (!g_encode) {
      cudaDriverEntryPointQueryResult q;
      void* fn = nullptr;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          q != cudaDriverEntryPointSuccess || fn == nullptr)
        return LORA_ECUDA;
      g_encode = reinterpret_cast<EncodeTiledFn>(fn);
    }
    d.ready = true;
  }
  if (!d.supported) return LORA_EDEVICE;
  *out = &d;
  return LORA_OK;
}

// 2-D bf16 tensor map over a row-major [outer, inner] matrix with row stride
// `ld` elements, 128-byte swizzle, zero fill outside the matrix.
int make_map(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer, uint64_t ld, uint32_t box_inner,
             uint32_t box_outer) {
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LORA_OK : LORA_ECUDA;
}

inline size_t up256(size_t x) { return (x + 255) & ~(size_t)255; }
inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline int cdiv(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }

int check_shape(const lora_shape* s) {
  if (!s) return LORA_ENULL;
  if (s->T < 8 || s->d_in < 8 || s->d_out < 8) return LORA_EINVAL;
  if ((s->T % 8) || (s->d_in % 8) || (s->d_out % 8)) return LORA_EINVAL;
  if (s->T > (1ll << 30) || s->d_in > (1ll << 20) || s->d_out > (1ll << 20)) return LORA_EINVAL;
  if (s->rank < 1 || s->rank > 128) return LORA_EINVAL;
  if (!isfinite(s->scale)) return LORA_EINVAL;
  return LORA_OK;
}

// Workspace regions of one projection.
struct Ws {
  size_t su_pad = 0, b_pad = 0, sv = 0;
  size_t total = 0;
};

Ws plan_ws(const lora_shape& s, int mode) {
  Ws w;
  const int64_t T = s.T, N = s.d_out, r8 = rank_pad8((int)s.rank);
  const bool pad = (s.rank % 8) != 0;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += up256(bytes);
    return o;
  };
  w.su_pad = take((size_t)T * r8 * 2);
  if (pad) w.b_pad = take((size_t)N * r8 * 2);
  if (mode & LORA_BWD) w.sv = take((size_t)T * r8 * 2);
  w.total = off;
  return w;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<uint8_t*>(ws) + off);
}

typedef __nv_bfloat16 bf;
inline const bf* cb(const lora_bf16* p) { return reinterpret_cast<const bf*>(p); }
inline bf* mb(lora_bf16* p) { return reinterpret_cast<bf*>(p); }

// Adapter operands of one projection's fused contraction.
struct Operands {
  const bf* s_in;  // su (forward) or sv (backward): [T, r], row stride ld_s
  int ld_s;
  const bf* B;     // forward: B [N, r], row stride ld_b
  int ld_b;
};

// Appends block (W, ldw, rw) -> (out, out2) to the row problem of activation X,
// opening a new problem when X differs or the concatenated rank would pass 128.
void add_row_block(std::vector<RowProb>& probs, const bf* X, int ldx, int T, int C, float scale, const bf* W,
                   int ldw, int rw, bf* out, int ld_out, bf* out2, int ld_out2, bool fuse) {
  RowProb* p = nullptr;
  if (fuse) {
    for (RowProb& q : probs) {
      int used = 0;
      for (int b = 0; b < q.nblk; ++b) used += rank_pad8(q.rw[b]);
      if (q.X == X && q.T == T && q.C == C && q.ldx == ldx && q.scale == scale && q.nblk < kMaxRankBlocks &&
          used + rank_pad8(rw) <= 128) {
        p = &q;
        break;
      }
    }
  }
  if (!p) {
    RowProb q;
    memset(&q, 0, sizeof(q));
    q.X = X;
    q.ldx = ldx;
    q.T = T;
    q.C = C;
    q.scale = scale;
    probs.push_back(q);
    p = &probs.back();
  }
  const int b = p->nblk++;
  p->W[b] = W;
  p->ldw[b] = ldw;
  p->rw[b] = rw;
  p->out[b] = out;
  p->ld_out[b] = ld_out;
  p->out2[b] = out2;
  p->ld_out2[b] = ld_out2;
}

void add_col_block(std::vector<ColProb>& probs, const bf* X, int ldx, int T, int C, const bf* S, int lds, int rs,
                   float* out, int out_cr, bool fuse) {
  ColProb* p = nullptr;
  if (fuse) {
    for (ColProb& q : probs) {
      int used = 0;
      for (int b = 0; b < q.nblk; ++b) used += rank_pad8(q.rs[b]);
      if (q.X == X && q.T == T && q.C == C && q.ldx == ldx && q.out_cr == out_cr && q.nblk < kMaxRankBlocks &&
          used + rank_pad8(rs) <= 128) {
        p = &q;
        break;
      }
    }
  }
  if (!p) {
    ColProb q;
    memset(&q, 0, sizeof(q));
    q.X = X;
    q.ldx = ldx;
    q.T = T;
    q.C = C;
    q.out_cr = out_cr;
    probs.push_back(q);
    p = &probs.back();
  }
  const int b = p->nblk++;
  p->S[b] = S;
  p->lds[b] = lds;
  p->rs[b] = rs;
  p->out[b] = out;
}

int launch_rows(std::vector<RowProb>& probs, bool w_rc, int num_sms, cudaStream_t st) {
  const int tile = rank_tile();
  for (size_t i0 = 0; i0 < probs.size(); i0 += kMaxRankProblems) {
    RowBatch b;
    memset(&b, 0, sizeof(b));
    int rmax = 16, max_chunks = 1;
    for (size_t i = i0; i < probs.size() && i < i0 + kMaxRankProblems; ++i) {
      RowProb& p = probs[i];
      int used = 0;
      for (int k = 0; k < p.nblk; ++k) used += rank_pad8(p.rw[k]);
      p.rpad = rank_pad16(used);
      rmax = std::max(rmax, p.rpad);
      max_chunks = std::max(max_chunks, cdiv(p.C, tile));
      p.tile_begin = b.tiles;
      b.tiles += cdiv(p.T, tile);
      b.p[b.n++] = p;
    }
    b.splits = rank_splits(b.tiles, max_chunks, num_sms);
    b.w_rc = w_rc ? 1 : 0;
    for (int i = 0; i < b.n; ++i) b.p[i].cps = cdiv(cdiv(b.p[i].C, tile), b.splits);
    if (launch_rowprod(b, rmax, st) != cudaSuccess) return LORA_ECUDA;
  }
  return LORA_OK;
}

int launch_cols(std::vector<ColProb>& probs, int num_sms, cudaStream_t st) {
  const int tile = rank_tile();
  for (size_t i0 = 0; i0 < probs.size(); i0 += kMaxRankProblems) {
    ColBatch b;
    memset(&b, 0, sizeof(b));
    int rmax = 16, max_chunks = 1;
    for (size_t i = i0; i < probs.size() && i < i0 + kMaxRankProblems; ++i) {
      ColProb& p = probs[i];
      int used = 0;
      for (int k = 0; k < p.nblk; ++k) used += rank_pad8(p.rs[k]);
      p.rpad = rank_pad16(used);
      rmax = std::max(rmax, p.rpad);
      max_chunks = std::max(max_chunks, cdiv(p.T, tile));
      p.tile_begin = b.tiles;
      b.tiles += cdiv(p.C, tile);
      b.p[b.n++] = p;
    }
    b.splits = rank_splits(b.tiles, max_chunks, num_sms);
    for (int i = 0; i < b.n; ++i) b.p[i].cps = cdiv(cdiv(b.p[i].T, tile), b.splits);
    if (launch_colprod(b, rmax, st) != cudaSuccess) return LORA_ECUDA;
  }
  return LORA_OK;
}

// ------------------------------------------------------------------ forward
// CTA pairs per cluster for a batch of fused contractions over tokens T_i:
// two pairs (weight tile shared) unless stacking 512 rows would waste work.
int choose_pairs(const std::vector<int64_t>& Ts) {
  for (int64_t T : Ts) {
    const int64_t rows1 = (T + 255) / 256 * 256, rows2 = (T + 511) / 512 * 512;
    if (rows2 * 100 > rows1 * 107) return 1;
  }
  return 2;
}

int add_fwd_problem(GemmBatch& b, const lora_proj& p, const Operands& o, int pairs) {
  const lora_shape& s = p.shape;
  const int i = b.num_problems;
  const int64_t T = s.T, K = s.d_in, N = s.d_out, r = s.rank;
  int rc;
  // activation boxes: one CTA's 128 rows x 64 contraction elements; weight
  // boxes: 64 rows x 64 (two per CTA, shared between the pairs of a cluster)
  if ((rc = make_map(&b.tmA[i], p.x, K, T, K, 64, 128)) != LORA_OK) return rc;
  if ((rc = make_map(&b.tmA2[i], o.s_in, r, T, o.ld_s, 64, 128)) != LORA_OK) return rc;
  if ((rc = make_map(&b.tmB[i], p.W, K, N, K, 64, 64)) != LORA_OK) return rc;
  if ((rc = make_map(&b.tmB2[i], o.B, r, N, o.ld_b, 64, 64)) != LORA_OK) return rc;
  GemmProblem& g = b.prob[i];
  g.out = mb(p.y);
  g.ldo = (int)N;
  g.M = (int)T;
  g.N = (int)N;
  g.Kmain = (int)K;
  g.r = (int)r;
  g.num_n_tiles = cdiv(N, gemm_tile_n());
  g.num_m_tiles = cdiv(T, (int64_t)gemm_tile_m() * pairs);
  g.m_fast = N >= T ? 1 : 0;  // weight operand [N, K] at least as large as x [T, K]
  g.kb_main = cdiv(K, gemm_tile_k());
  g.kb_total = g.kb_main + cdiv(r, gemm_tile_k());
  g.tile_begin = b.total_tiles;
  b.total_tiles += g.num_m_tiles * g.num_n_tiles;
  b.num_problems++;
  return LORA_OK;
}

// ------------------------------------------------------------------ backward
int add_bwd_problem(GemmBatch& b, const lora_proj& p, const Operands& o, int pairs) {
  const lora_shape& s = p.shape;
  const int i = b.num_problems;
  const int64_t T = s.T, K = s.d_in, N = s.d_out, r = s.rank;
  int rc;
  if ((rc = make_map(&b.tmA[i], p.dy, N, T, N, 64, 128)) != LORA_OK) return rc;
  if ((rc = make_map(&b.tmA2[i], o.s_in, r, T, o.ld_s, 64, 128)) != LORA_OK) return rc;
  // W [N, K] read MN-major: inner dimension K (the GEMM's output columns), rows = contraction
  if ((rc = make_map(&b.tmB[i], p.W, K, N, K, 64, 64)) != LORA_OK) return rc;
  if ((rc = make_map(&b.tmB2[i], p.A, K, r, K, 64, 64)) != LORA_OK) return rc;
  GemmProblem& g = b.prob[i];
  g.out = mb(p.dx);
  g.ldo = (int)K;
  g.M = (int)T;
  g.N = (int)K;
  g.Kmain = (int)N;
  g.r = (int)r;
  g.num_n_tiles = cdiv(K, gemm_tile_n());
  g.num_m_tiles = cdiv(T, (int64_t)gemm_tile_m() * pairs);
  g.m_fast = K >= T ? 1 : 0;  // weight operand [N, K] at least as large as dy [T, N]
  g.kb_main = cdiv(N, gemm_tile_k());
  g.kb_total = g.kb_main + cdiv(r, gemm_tile_k());
  g.tile_begin = b.total_tiles;
  b.total_tiles += g.num_m_tiles * g.num_n_tiles;
  b.num_problems++;
  return LORA_OK;
}

void init_batch(GemmBatch& b, const DeviceInfo* d) {
  memset(&b, 0, sizeof(b));
  b.status = d->status;
  b.limit_ns = g_wait_limit_ns;
}

// ------------------------------------------------------------------ checks
int check_fwd_ptrs(const lora_proj& p) {
  if (!p.x || !p.W || !p.A || !p.B || !p.y) return LORA_ENULL;
  const void* ps[] = {p.x, p.W, p.A, p.B, p.y, p.su};
  for (const void* q : ps)
    if (q && !aligned16(q)) return LORA_EALIGN;
  return LORA_OK;
}

int check_bwd_ptrs(const lora_proj& p) {
  if (!p.dy || !p.x || !p.W || !p.A || !p.B || !p.su || !p.dA || !p.dB) return LORA_ENULL;
  const void* ps[] = {p.dy, p.x, p.W, p.A, p.B, p.su, p.dx, p.dA, p.dB};
  for (const void* q : ps)
    if (q && !aligned16(q)) return LORA_EALIGN;
  return LORA_OK;
}

int check_ws(void* ws, size_t ws_bytes, size_t need) {
  if (!ws || ws_bytes < need) return LORA_EWORKSPACE;
  if (reinterpret_cast<uintptr_t>(ws) & 255u) return LORA_EALIGN;
  return LORA_OK;
}

// Runs the given projections in `mode`; every argument already validated.
int run_step(const lora_proj* projs, int n, int mode, void* ws, const std::vector<Ws>& plans,
             const std::vector<size_t>& offs, DeviceInfo* d, cudaStream_t st) {
  int rc;
  auto W_ = [&](int i) { return at<uint8_t>(ws, offs[i]); };
  // tile counters of the fused-GEMM launches live in the workspace header
  int* counters = at<int>(ws, 0);
  int next_counter = 0;
  if (cudaMemsetAsync(counters, 0, kWsHeader, st) != cudaSuccess) return LORA_ECUDA;
  if (mode & LORA_FWD) {
    std::vector<Operands> ops(n);
    std::vector<RowProb> rows;
    {
      ProfScope ps(LORA_KERNEL_PAD, st);
      for (int i = 0; i < n; ++i) {
        const lora_proj& p = projs[i];
        const int T = (int)p.shape.T, K = (int)p.shape.d_in, N = (int)p.shape.d_out, r = (int)p.shape.rank;
        const int r8 = rank_pad8(r);
        const bool pad = (r % 8) != 0;
        bf* su_gemm = (p.su && !pad) ? mb(p.su) : at<bf>(W_(i), plans[i].su_pad);
        const int ld_gemm = (p.su && !pad) ? r : r8;
        bf* su_user2 = (p.su && pad) ? mb(p.su) : nullptr;
        add_row_block(rows, cb(p.x), K, T, K, p.shape.scale, cb(p.A), K, r, su_gemm, ld_gemm, su_user2, r, true);
        ops[i].s_in = su_gemm;
        ops[i].ld_s = ld_gemm;
        if (pad) {
          if (launch_pad_cols(cb(p.B), N, r, at<bf>(W_(i), plans[i].b_pad), r8, st) != cudaSuccess)
            return LORA_ECUDA;
          ops[i].B = at<bf>(W_(i), plans[i].b_pad);
          ops[i].ld_b = r8;
        } else {
          ops[i].B = cb(p.B);
          ops[i].ld_b = r;
        }
      }
    }
    {
      ProfScope ps(LORA_KERNEL_ROWPROJ, st);
      if ((rc = launch_rows(rows, true, d->num_sms, st)) != LORA_OK) return rc;
    }
    // heavier problems first so that the static tile walk ends balanced
    std::vector<int> order(n);
    for (int i = 0; i < n; ++i) order[i] = i;
    std::stable_sort(order.begin(), order.end(),
                     [&](int a, int b) { return projs[a].shape.d_in > projs[b].shape.d_in; });
    for (int i0 = 0; i0 < n; i0 += kMaxProblems) {
      GemmBatch b;
      init_batch(b, d);
      b.tile_counter = counters + next_counter++;
      std::vector<int64_t> Ts;
      for (int i = i0; i < n && i < i0 + kMaxProblems; ++i) Ts.push_back(projs[order[i]].shape.T);
      const int pairs = choose_pairs(Ts);
      for (int i = i0; i < n && i < i0 + kMaxProblems; ++i)
        if ((rc = add_fwd_problem(b, projs[order[i]], ops[order[i]], pairs)) != LORA_OK) return rc;
      ProfScope ps(LORA_KERNEL_GEMM_FWD, st);
      if (launch_fused_gemm(b, false, pairs, d->num_sms, st) != cudaSuccess) return LORA_ECUDA;
    }
  }
  if (mode & LORA_BWD) {
    std::vector<Operands> ops(n);
    std::vector<RowProb> rows;
    std::vector<ColProb> cols;
    std::vector<const bf*> su_in(n);
    std::vector<int> ld_su(n);
    {
      ProfScope ps(LORA_KERNEL_PAD, st);
      for (int i = 0; i < n; ++i) {
        const lora_proj& p = projs[i];
        const int T = (int)p.shape.T, N = (int)p.shape.d_out, r = (int)p.shape.rank, r8 = rank_pad8(r);
        const bool pad = (r % 8) != 0;
        const bf* B_in = cb(p.B);
        int ld_b = r;
        su_in[i] = cb(p.su);
        ld_su[i] = r;
        if (pad) {
          if (launch_pad_cols(cb(p.su), T, r, at<bf>(W_(i), plans[i].su_pad), r8, st) != cudaSuccess ||
              launch_pad_cols(cb(p.B), N, r, at<bf>(W_(i), plans[i].b_pad), r8, st) != cudaSuccess)
            return LORA_ECUDA;
          su_in[i] = at<bf>(W_(i), plans[i].su_pad);
          ld_su[i] = r8;
          B_in = at<bf>(W_(i), plans[i].b_pad);
          ld_b = r8;
        }
        bf* sv = at<bf>(W_(i), plans[i].sv);
        add_row_block(rows, cb(p.dy), N, T, N, p.shape.scale, B_in, ld_b, r, sv, r8, nullptr, 0, false);
        ops[i].s_in = sv;
        ops[i].ld_s = r8;
      }
    }
    {
      ProfScope ps(LORA_KERNEL_ROWPROJ, st);
      if ((rc = launch_rows(rows, false, d->num_sms, st)) != LORA_OK) return rc;
    }
    for (int i = 0; i < n; ++i) {
      const lora_proj& p = projs[i];
      const int T = (int)p.shape.T, K = (int)p.shape.d_in, N = (int)p.shape.d_out, r = (int)p.shape.rank;
      add_col_block(cols, cb(p.dy), N, T, N, su_in[i], ld_su[i], r, p.dB, 1, false);
    }
    for (int i = 0; i < n; ++i) {
      const lora_proj& p = projs[i];
      const int T = (int)p.shape.T, K = (int)p.shape.d_in, r = (int)p.shape.rank;
      add_col_block(cols, cb(p.x), K, T, K, ops[i].s_in, ops[i].ld_s, r, p.dA, 0, true);
    }
    {
      ProfScope ps(LORA_KERNEL_COLPROJ, st);
      if ((rc = launch_cols(cols, d->num_sms, st)) != LORA_OK) return rc;
    }
    std::vector<int> order;
    for (int i = 0; i < n; ++i)
      if (projs[i].dx) order.push_back(i);
    std::stable_sort(order.begin(), order.end(),
                     [&](int a, int b) { return projs[a].shape.d_out > projs[b].shape.d_out; });
    for (size_t i0 = 0; i0 < order.size(); i0 += kMaxProblems) {
      GemmBatch b;
      init_batch(b, d);
      b.tile_counter = counters + next_counter++;
      std::vector<int64_t> Ts;
      for (size_t i = i0; i < order.size() && i < i0 + kMaxProblems; ++i) Ts.push_back(projs[order[i]].shape.T);
      const int pairs = choose_pairs(Ts);
      for (size_t i = i0; i < order.size() && i < i0 + kMaxProblems; ++i)
        if ((rc = add_bwd_problem(b, projs[order[i]], ops[order[i]], pairs)) != LORA_OK) return rc;
      ProfScope ps(LORA_KERNEL_GEMM_BWD, st);
      if (launch_fused_gemm(b, true, pairs, d->num_sms, st) != cudaSuccess) return LORA_ECUDA;
    }
  }
  return LORA_OK;
}

int plan_all(const lora_proj* projs, int n, int mode, int num_sms, std::vector<Ws>* plans,
             std::vector<size_t>* offs, size_t* total) {
  size_t off = kWsHeader;
  plans->resize(n);
  offs->resize(n);
  for (int i = 0; i < n; ++i) {
    int rc = check_shape(&projs[i].shape);
    if (rc != LORA_OK) return rc;
    (*plans)[i] = plan_ws(projs[i].shape, mode);
    (*offs)[i] = off;
    off += up256((*plans)[i].total);
  }
  *total = off;
  return LORA_OK;
}

}  // namespace

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

}  // namespace lora

using namespace lora;

extern "C" {

int lora_version(void) { return 100; }

const char* lora_strerror(int code) {
  switch (code) {
    case LORA_OK: return "ok";
    case LORA_EINVAL: return "invalid shape, rank, scale, mode or count";
    case LORA_ENULL: return "required pointer is NULL";
    case LORA_EALIGN: return "pointer not 16-byte aligned (workspace: 256-byte)";
    case LORA_ECUDA: return "CUDA runtime call or kernel launch failed";
    case LORA_ETIMEOUT: return "a device-side bounded wait expired";
    case LORA_EWORKSPACE: return "workspace missing or too small";
    case LORA_EDEVICE: return "current device is not a compute capability 10.3 (GB300) GPU";
    default: return "unknown error";
  }
}

int lora_set_wait_limit_ns(int64_t ns) {
  std::lock_guard<std::mutex> lk(g_mu);
  g_wait_limit_ns = ns > 0 ? (long long)ns : kDefaultWaitNs;
  return LORA_OK;
}

int lora_workspace_size(const lora_shape* shape, int mode, size_t* bytes) {
  if (!shape || !bytes) return LORA_ENULL;
  if (mode < LORA_FWD || mode > LORA_FWD_BWD) return LORA_EINVAL;
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  return lora_stack_workspace_size(&p, 1, mode, bytes);
}

int lora_stack_workspace_size(const lora_proj* projs, int n_proj, int mode, size_t* bytes) {
  if (!projs || !bytes) return LORA_ENULL;
  if (n_proj < 1 || n_proj > 64 || mode < LORA_FWD || mode > LORA_FWD_BWD) return LORA_EINVAL;
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != LORA_OK) return rc;
  std::vector<Ws> plans;
  std::vector<size_t> offs;
  return plan_all(projs, n_proj, mode, d->num_sms, &plans, &offs, bytes);
}

int lora_stack_step(const lora_proj* projs, int n_proj, int mode, void* workspace, size_t workspace_bytes,
                    void* stream) {
  if (!projs) return LORA_ENULL;
  if (n_proj < 1 || n_proj > 64 || mode < LORA_FWD || mode > LORA_FWD_BWD) return LORA_EINVAL;
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != LORA_OK) return rc;
  std::vector<Ws> plans;
  std::vector<size_t> offs;
  size_t need = 0;
  if ((rc = plan_all(projs, n_proj, mode, d->num_sms, &plans, &offs, &need)) != LORA_OK) return rc;
  for (int i = 0; i < n_proj; ++i) {
    if ((mode & LORA_FWD) && (rc = check_fwd_ptrs(projs[i])) != LORA_OK) return rc;
    if ((mode & LORA_BWD) && (rc = check_bwd_ptrs(projs[i])) != LORA_OK) return rc;
    if (mode == LORA_FWD_BWD && !projs[i].su) return LORA_ENULL;  // the backward needs the saved su
  }
  if ((rc = check_ws(workspace, workspace_bytes, need)) != LORA_OK) return rc;
  return run_step(projs, n_proj, mode, workspace, plans, offs, d, static_cast<cudaStream_t>(stream));
}

int lora_linear_fwd(const lora_shape* shape, const lora_bf16* x, const lora_bf16* W, const lora_bf16* A,
                    const lora_bf16* B, lora_bf16* y, lora_bf16* su, void* workspace, size_t workspace_bytes,
                    void* stream) {
  if (!shape) return LORA_ENULL;
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  p.x = x;
  p.W = W;
  p.A = A;
  p.B = B;
  p.y = y;
  p.su = su;
  return lora_stack_step(&p, 1, LORA_FWD, workspace, workspace_bytes, stream);
}

int lora_linear_bwd(const lora_shape* shape, const lora_bf16* dy, const lora_bf16* x, const lora_bf16* W,
                    const lora_bf16* A, const lora_bf16* B, const lora_bf16* su, lora_bf16* dx, float* dA,
                    float* dB, void* workspace, size_t workspace_bytes, void* stream) {
  if (!shape) return LORA_ENULL;
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  p.dy = dy;
  p.x = x;
  p.W = W;
  p.A = A;
  p.B = B;
  p.su = const_cast<lora_bf16*>(su);  // read only in the backward
  p.dx = dx;
  p.dA = dA;
  p.dB = dB;
  return lora_stack_step(&p, 1, LORA_BWD, workspace, workspace_bytes, stream);
}

int64_t lora_launch_count(void) { return (int64_t)g_launches.load(); }

int lora_profile_begin(void) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof.recs.clear();
  g_prof.next = 0;
  g_prof.on = true;
  return LORA_OK;
}

int lora_profile_end(double* ms, int64_t* launches) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (!g_prof.on) return LORA_EINVAL;
  double acc[LORA_KERNEL_KINDS] = {0};
  int64_t cnt[LORA_KERNEL_KINDS] = {0};
  int rc = LORA_OK;
  for (const ProfRec& r : g_prof.recs) {
    float t = 0.f;
    if (cudaEventSynchronize(r.b) != cudaSuccess || cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) {
      rc = LORA_ECUDA;
      continue;
    }
    acc[r.kind] += t;
    cnt[r.kind] += r.launches;
  }
  for (int k = 0; k < LORA_KERNEL_KINDS; ++k) {
    if (ms) ms[k] = acc[k];
    if (launches) launches[k] = cnt[k];
  }
  g_prof.recs.clear();
  g_prof.next = 0;
  g_prof.on = false;
  return rc;
}

int lora_read_status(void* stream, int* status, int reset) {
  if (!status) return LORA_ENULL;
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return LORA_ECUDA;
  int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_status, sizeof(int)) != cudaSuccess) return LORA_ECUDA;
  if (reset) {
    const int z = 0;
    if (cudaMemcpyToSymbol(g_status, &z, sizeof(int)) != cudaSuccess) return LORA_ECUDA;
  }
  *status = v ? LORA_ETIMEOUT : LORA_OK;
  return LORA_OK;
}

}  // extern "C"
