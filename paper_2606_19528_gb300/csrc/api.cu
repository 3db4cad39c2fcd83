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
#include <cstdlib>
#include <functional>
#include <map>
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
  uint32_t mask = 0;  // kinds bracketed with events
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
    if (!g_prof.on || !((g_prof.mask >> kind) & 1u)) return;
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

// 2-D bf16 (or fp32) tensor map over a row-major [outer, inner] matrix with
// row stride `ld` elements, 128-byte swizzle, zero fill outside the matrix.
int make_map(CUtensorMap* m, const void* ptr, uint64_t inner, uint64_t outer, uint64_t ld, uint32_t box_inner,
             uint32_t box_outer, bool f32 = false) {
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * (f32 ? 4 : 2)};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? LORA_OK : LORA_ECUDA;
}

// 2-D tensor map of `dtype` elements over a row-major [outer, inner] matrix
// with row stride `ld` elements, no swizzle (staging boxes read by threads).
int make_map_plain(CUtensorMap* m, CUtensorMapDataType dtype, int esize, const void* ptr, uint64_t inner,
                   uint64_t outer, uint64_t ld, uint32_t box_inner, uint32_t box_outer) {
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {ld * (uint64_t)esize};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, dtype, 2, const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
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
  if (s->rank < 0 || s->rank > 128) return LORA_EINVAL;  // rank 0: frozen projection, no adapter
  if (!isfinite(s->scale)) return LORA_EINVAL;
  return LORA_OK;
}

// Workspace regions of one projection.
struct Ws {
  size_t su_pad = 0, b_pad = 0, sv = 0, bt = 0, sut = 0, svt = 0;
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
  if (mode & LORA_BWD) {
    w.sv = take((size_t)T * r8 * 2);
    w.bt = take((size_t)N * r8 * 2);   // B^T, zero rows past r
    w.sut = take((size_t)T * r8 * 2);  // su^T, zero rows past r
    w.svt = take((size_t)T * r8 * 2);  // sv^T, zero rows past r
  }
  w.total = off;
  return w;
}

// Workspace of a call: [GEMM tile counters | rank-r partials |
// per-projection regions]; the counters are cleared by one memset at the
// start of a call.
// The rank-r arenas are sized for the projections without input sharing,
// an upper bound of what grouped problems need (a group's padded rank is at
// most the sum of its members').
enum { kPhFwdRows = 0, kPhBwdRows = 1, kPhBwdCols = 2, kPhases = 3 };

struct Plan {
  std::vector<Ws> ws;
  std::vector<size_t> offs;
  size_t part_off[kPhases] = {0, 0, 0}, n_partials[kPhases] = {0, 0, 0};
  // split contractions: per projection, the split counts of its forward and
  // backward contraction and its fp32 partial buffer (planned from the shapes)
  std::vector<int> split_f, split_b;
  std::vector<size_t> split_off;
  size_t zero_bytes = 0;  // [0, zero_bytes) is cleared at the start of a call
  size_t total = 0;
  // the fused passes over dy cut for the whole device, as a backward call cuts them, even where a
  // side stream runs them on a few SMs (the checkpointed stack, whose re-forward-and-backward calls
  // must sum sv and dB exactly as the saved schedule's backward calls)
  bool dy_cut_device = false;
};

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<uint8_t*>(ws) + off);
}

typedef __nv_bfloat16 bf;
inline const bf* cb(const lora_bf16* p) { return reinterpret_cast<const bf*>(p); }
inline bf* mb(lora_bf16* p) { return reinterpret_cast<bf*>(p); }

inline bool is_q4(const lora_proj& p) { return p.Wq.codes != nullptr; }
inline int64_t rup(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// ------------------------------------------------------------------ fused-contraction problems
// Output [M, N] over a contraction of Kc base columns plus an r-wide adapter
// slab; one contraction pass, output written directly (no split).
// tile_n: the launch's tile width (gemm_tile_n(), or gemm_tile_n_f32() for fp32 output).
void gemm_shape(GemmProblem& g, int64_t M, int64_t N, int64_t Kc, int64_t r, int tile_n = 0) {
  g.ldo = (int)N;
  g.out_f32 = 0;
  g.M = (int)M;
  g.N = (int)N;
  g.Kmain = (int)Kc;
  g.r = (int)r;
  g.num_n_tiles = cdiv(N, tile_n > 0 ? tile_n : gemm_tile_n());
  g.num_m_tiles = cdiv(M, gemm_tile_m());
  g.m_fast = N >= M ? 1 : 0;  // the weight operand at least as large as the activation operand
  g.kb_main = cdiv(Kc, gemm_tile_k());
  g.kb_total = g.kb_main + cdiv(r, gemm_tile_k());
  g.splits = 1;
  g.kb_split = g.kb_total;
  g.m_pad = g.num_m_tiles * gemm_tile_m();
  g.part = nullptr;
  g.ldp = 0;
  g.lse = nullptr;
  g.ld_lse = 0;
  g.tau = nullptr;
  g.cnt = nullptr;
  g.cand = nullptr;
  g.cap = 0;
  g.row_off = g.col_off = g.sym = 0;
}

// Appends the problem just filled in at b.prob[b.num_problems].
void add_problem(GemmBatch& b) {
  GemmProblem& g = b.prob[b.num_problems];
  g.tile_begin = b.total_tiles;
  b.total_tiles += g.num_m_tiles * g.num_n_tiles * g.splits;
  b.num_problems++;
}

constexpr int kPlanSms = 152;              // SMs the split rule plans for (a GB300)
constexpr int kPlanPairs = kPlanSms / 2;  // CTA pairs of a launch on all of them

// Split contraction for batches with fewer output tiles than CTA pairs.  The
// persistent kernel hands out (tile, split) units in order to whichever pair
// is free, so for each candidate split length L (problem p cut into
// ceil(kb_p / L) splits, at most 8) the walk is simulated on `pairs` pairs in
// units of one k-block of a 256 x 512 tile (~0.77 us at the measured rate),
// with a fixed cost per unit (pipeline fill, epilogue), one more for an fp32
// partial epilogue, and the reduce launch plus its traffic; the cheapest
// candidate wins (fewer splits on ties).  Choices are cached per shape set.
constexpr double kUnitFixBlocks = 3.0;    // per unit: pipeline fill and epilogue
constexpr double kPartEpiBlocks = 1.0;    // per split unit: fp32 partial tile instead of bf16
constexpr double kReduceFixBlocks = 6.0;  // the reduce launch
constexpr double kBytesPerBlock = 5.0e6;  // HBM bytes moved in one block time

double simulate_splits(const GemmBatch& b, const int* sp, int pairs) {
  std::vector<double> fin(pairs, 0.0);  // min-heap of pair finish times
  std::make_heap(fin.begin(), fin.end(), std::greater<double>());
  double reduce = 0.0;
  bool any = false;
  for (int p = 0; p < b.num_problems; ++p) {
    const GemmProblem& g = b.prob[p];
    const int per = g.num_m_tiles * g.num_n_tiles;
    const int kbs = (g.kb_total + sp[p] - 1) / sp[p];
    for (int ks = 0; ks < sp[p]; ++ks) {
      const int len = std::min(g.kb_total, (ks + 1) * kbs) - ks * kbs;
      const double d = len + kUnitFixBlocks + (sp[p] > 1 ? kPartEpiBlocks : 0.0);
      for (int t = 0; t < per; ++t) {
        std::pop_heap(fin.begin(), fin.end(), std::greater<double>());
        fin.back() += d;
        std::push_heap(fin.begin(), fin.end(), std::greater<double>());
      }
    }
    if (sp[p] > 1) {
      any = true;
      reduce += (double)g.m_pad * g.N * (4.0 * sp[p] + 2.0) / kBytesPerBlock;
    }
  }
  return *std::max_element(fin.begin(), fin.end()) + reduce + (any ? kReduceFixBlocks : 0.0);
}

void choose_splits(const GemmBatch& b, int* splits, int pairs = kPlanPairs) {
  long long tiles = 0;
  std::vector<long long> key;
  key.push_back(pairs);
  for (int p = 0; p < b.num_problems; ++p) {
    const GemmProblem& g = b.prob[p];
    tiles += (long long)g.num_m_tiles * g.num_n_tiles;
    key.insert(key.end(), {g.num_m_tiles, g.num_n_tiles, g.kb_total, g.m_pad, g.N});
    splits[p] = 1;
  }
  if (tiles == 0 || tiles >= pairs) return;
  static std::mutex mu;
  static std::map<std::vector<long long>, std::vector<int>> cache;
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      std::copy(it->second.begin(), it->second.end(), splits);
      return;
    }
  }
  std::vector<int> cand;
  for (int p = 0; p < b.num_problems; ++p)
    for (int s = 1; s <= 8; ++s) cand.push_back((b.prob[p].kb_total + s - 1) / s);
  std::sort(cand.begin(), cand.end(), std::greater<int>());  // longest splits (fewest) first
  cand.erase(std::unique(cand.begin(), cand.end()), cand.end());
  std::vector<int> sp(b.num_problems), best(b.num_problems, 1);
  double best_cost = simulate_splits(b, best.data(), pairs);
  for (int L : cand) {
    for (int p = 0; p < b.num_problems; ++p) {
      const int kb = b.prob[p].kb_total;
      int s = std::min(8, std::max(1, (kb + L - 1) / L));
      if (s > 1) s = (kb + (kb + s - 1) / s - 1) / ((kb + s - 1) / s);  // no empty split
      sp[p] = s;
    }
    const double c = simulate_splits(b, sp.data(), pairs);
    if (c < best_cost - 1e-9) {
      best_cost = c;
      best = sp;
    }
  }
  std::copy(best.begin(), best.end(), splits);
  std::lock_guard<std::mutex> lk(mu);
  if (cache.size() > 4096) cache.clear();
  cache.emplace(key, best);
}

// Cluster split for launches with too few output tiles to fill the GPU: when
// the batch's 256 x 512 tiles number fewer than the launch's CTA pairs and
// its 256 x 256 tiles, two pairs each, fit on them (and all at once on the
// device), each tile goes to a cluster of two CTA pairs that contract one half
// of its blocks each and sum the halves through distributed shared memory: no
// fp32 partials in memory and no reduce launch.  Problems of fewer than
// kCsMinBlocks blocks are not worth cutting; beyond kCsMaxBlocks the partials
// cost little next to the contraction, and the wide tiles of the split into
// partials contract faster than the cluster's 256 x 256 tiles (LM-head dh
// contraction over the full vocabulary, 2004 blocks: 0.96 against 0.91 ms).
// Rewrites the batch's tile list for 256-column tiles and returns true when
// it applies.
constexpr int kCsMinBlocks = 8;
constexpr int kCsMaxBlocks = 256;

bool use_cluster_split(GemmBatch& b, bool b_mn, int pairs) {
  long long wide = 0, narrow = 0;
  for (int p = 0; p < b.num_problems; ++p) {
    const GemmProblem& g = b.prob[p];
    if (g.kb_total < kCsMinBlocks || g.kb_total > kCsMaxBlocks || g.out_f32) return false;
    wide += (long long)g.num_m_tiles * g.num_n_tiles;
    narrow += (long long)g.num_m_tiles * cdiv(g.N, gemm_tile_n_f32());
  }
  if (wide == 0 || wide >= pairs || 2 * narrow > pairs) return false;
  if (narrow > gemm_cs_max_clusters(b_mn)) return false;
  b.total_tiles = 0;
  for (int p = 0; p < b.num_problems; ++p) {
    GemmProblem& g = b.prob[p];
    g.num_n_tiles = cdiv(g.N, gemm_tile_n_f32());
    g.splits = 1;
    g.kb_split = g.kb_total;
    g.tile_begin = b.total_tiles;
    b.total_tiles += g.num_m_tiles * g.num_n_tiles;
  }
  return true;
}

// fp32 partial elements of a problem cut into `sp` splits.
size_t split_floats(const GemmProblem& g, int sp) {
  return sp > 1 ? up256((size_t)sp * g.m_pad * (size_t)rup(g.N, 4) * 4) / 4 : 0;
}

// Applies split counts (partials of problem p at parts[p]): tile list, and
// fp32 output maps over the partial buffers.
int apply_splits(GemmBatch& b, const int* splits, float* const* parts) {
  b.total_tiles = 0;
  for (int p = 0; p < b.num_problems; ++p) {
    GemmProblem& g = b.prob[p];
    if (splits[p] > 1) {
      g.splits = splits[p];
      g.kb_split = (g.kb_total + g.splits - 1) / g.splits;
      g.ldp = (int)rup(g.N, 4);
      g.part = parts[p];
      const int rc = make_map(&b.tmOut[p], g.part, g.N, (uint64_t)g.splits * g.m_pad, g.ldp, 32, 32, true);
      if (rc != LORA_OK) return rc;
    }
    g.tile_begin = b.total_tiles;
    b.total_tiles += g.num_m_tiles * g.num_n_tiles * g.splits;
  }
  return LORA_OK;
}


// Adapter operands of one projection's fused contraction.
struct Operands {
  const bf* s_in;  // su (forward) or sv (backward): [T, r], row stride ld_s
  int ld_s;
  const bf* B;     // forward: B [N, r], row stride ld_b
  int ld_b;
};

// Host description of a rank-r problem before its tensor maps are encoded.
struct RowSpec {
  const bf* X;
  int ldx, T, C, nblk;
  float scale;
  const bf* W[kMaxRankBlocks];
  int ldw[kMaxRankBlocks], rw[kMaxRankBlocks];
  bf* out[kMaxRankBlocks];
  int ld_out[kMaxRankBlocks];
  bf* out2[kMaxRankBlocks];
  int ld_out2[kMaxRankBlocks];
  bf* outT[kMaxRankBlocks];
};
struct ColSpec {
  const bf* X;
  int ldx, T, C, nblk, out_cr;
  const bf* S[kMaxRankBlocks];
  int lds[kMaxRankBlocks], rs[kMaxRankBlocks];
  float* out[kMaxRankBlocks];
};

inline int used_rank(const int* r, int n) {
  int u = 0;
  for (int k = 0; k < n; ++k) u += rank_pad8(r[k]);
  return u;
}

// Appends block (W, ldw, rw) -> (out, out2, outT) to the row problem of
// activation X, opening a new problem when X differs or the concatenated rank
// would pass 128.
void add_row_block(std::vector<RowSpec>& probs, const bf* X, int ldx, int T, int C, float scale, const bf* W,
                   int ldw, int rw, bf* out, int ld_out, bf* out2, int ld_out2, bf* outT, bool fuse) {
  RowSpec* p = nullptr;
  if (fuse) {
    for (RowSpec& q : probs)
      if (q.X == X && q.T == T && q.C == C && q.ldx == ldx && q.scale == scale && q.nblk < kMaxRankBlocks &&
          used_rank(q.rw, q.nblk) + rank_pad8(rw) <= 128) {
        p = &q;
        break;
      }
  }
  if (!p) {
    RowSpec q;
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
  p->outT[b] = outT;
}

void add_col_block(std::vector<ColSpec>& probs, const bf* X, int ldx, int T, int C, const bf* S, int lds, int rs,
                   float* out, int out_cr, bool fuse) {
  ColSpec* p = nullptr;
  if (fuse) {
    for (ColSpec& q : probs)
      if (q.X == X && q.T == T && q.C == C && q.ldx == ldx && q.out_cr == out_cr && q.nblk < kMaxRankBlocks &&
          used_rank(q.rs, q.nblk) + rank_pad8(rs) <= 128) {
        p = &q;
        break;
      }
  }
  if (!p) {
    ColSpec q;
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

// fp32 partials of one rank-r phase.
struct Arena {
  float* partials;
  size_t n_partials;
};

constexpr int kMinUnitChunks = 8;  // smallest work unit (64-wide chunks); sizes the partial arenas

// Chunks per unit for a launch.  The persistent grid (max_ctas CTAs) takes
// units round-robin, so the launch lasts about ceil(units / CTAs) units; the
// cost of a size is that makespan in chunks, plus a fixed charge for the
// partial-sum pass when any tile needs several units.  Ties go to the larger
// unit (fewer partials).
template <typename Spec, typename LenFn>
int choose_unit_chunks(const std::vector<Spec>& specs, size_t i0, size_t i1, int max_ctas, LenFn len) {
  int best = kMinUnitChunks;
  long long best_cost = -1;
  for (int u : {64, 32, 16, 8}) {
    long long units = 0;
    bool partials = false;
    for (size_t i = i0; i < i1; ++i) {
      const auto tl = len(specs[i]);  // (tiles, reduction length)
      const long long upt = cdiv(cdiv(tl.second, 64), u);
      units += (long long)tl.first * upt;
      partials = partials || upt > 1;
    }
    const long long ctas = std::min<long long>(units, (long long)max_ctas);
    const long long cost = (units + ctas - 1) / ctas * u + (partials ? 4 : 0);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = u;
    }
  }
  return best;
}

// Row products of one phase on `ctas` persistent CTAs (one per SM).
int launch_rows(const std::vector<RowSpec>& specs, const Arena& ar, const DeviceInfo* d, int ctas, cudaStream_t st) {
  const int tile = rank_mma_tile();
  size_t pf = 0;
  int rc;
  for (size_t i0 = 0; i0 < specs.size(); i0 += kMaxRankProblems) {
    const size_t i1 = std::min(specs.size(), i0 + kMaxRankProblems);
    RowBatch b;
    memset(&b, 0, sizeof(b));
    b.tile_rows = tile;
    // one persistent CTA per SM; (tiles, reduction length) of a row problem
    b.unit_chunks = choose_unit_chunks(specs, i0, i1, ctas, [&](const RowSpec& q) {
      return std::make_pair(cdiv(q.T, tile), q.C);
    });
    int rmax = 16;
    for (size_t i = i0; i < i1; ++i) {
      const RowSpec& sp = specs[i];
      RowProb& p = b.p[b.n++];
      p.T = sp.T;
      p.C = sp.C;
      p.nblk = sp.nblk;
      p.scale = sp.scale;
      if ((rc = make_map(&p.tmX, sp.X, sp.C, sp.T, sp.ldx, 64, tile)) != LORA_OK) return rc;
      int bytes = tile * 64 * 2;
      for (int k = 0; k < sp.nblk; ++k) {
        p.rw[k] = sp.rw[k];
        p.out[k] = sp.out[k];
        p.ld_out[k] = sp.ld_out[k];
        p.out2[k] = sp.out2[k];
        p.ld_out2[k] = sp.ld_out2[k];
        p.outT[k] = sp.outT[k];
        const int r8 = rank_pad8(sp.rw[k]);
        // W_b [r_b, C]: 64 columns x r8 rows, rows past r_b zero-filled
        if ((rc = make_map(&p.tmW[k], sp.W[k], sp.C, sp.rw[k], sp.ldw[k], 64, r8)) != LORA_OK) return rc;
        bytes += 64 * r8 * 2;
      }
      p.tx_bytes = bytes;
      p.rpad = rank_pad16(used_rank(sp.rw, sp.nblk));
      rmax = std::max(rmax, p.rpad);
      const int tiles = cdiv(p.T, tile);
      p.upt = cdiv(cdiv(p.C, 64), b.unit_chunks);
      p.unit_begin = b.units;
      b.units += tiles * p.upt;
      p.part_off = (long long)pf;
      p.red_begin = b.red_total;
      if (p.upt > 1) {
        pf += (size_t)tiles * p.upt * tile * p.rpad;
        b.red_total += tiles * tile * p.rpad;
      }
    }
    if (pf > ar.n_partials) return LORA_EWORKSPACE;  // planning bound violated
    b.partials = ar.partials;
    b.status = d->status;
    b.limit_ns = g_wait_limit_ns;
    if (launch_rowmma(b, rmax, ctas, st) != cudaSuccess) return LORA_ECUDA;
  }
  return LORA_OK;
}

// Column products of one phase on `ctas` persistent CTAs (one per SM).
int launch_cols(const std::vector<ColSpec>& specs, const Arena& ar, const DeviceInfo* d, int ctas, cudaStream_t st) {
  const int tile = rank_mma_tile();
  size_t pf = 0;
  int rc;
  for (size_t i0 = 0; i0 < specs.size(); i0 += kMaxRankProblems) {
    const size_t i1 = std::min(specs.size(), i0 + kMaxRankProblems);
    ColBatch b;
    memset(&b, 0, sizeof(b));
    b.tile_rows = tile;
    // (tiles, reduction length) of a column problem
    b.unit_chunks = choose_unit_chunks(specs, i0, i1, ctas, [&](const ColSpec& q) {
      return std::make_pair(cdiv(q.C, tile), q.T);
    });
    int rmax = 16;
    for (size_t i = i0; i < i1; ++i) {
      const ColSpec& sp = specs[i];
      ColProb& p = b.p[b.n++];
      p.T = sp.T;
      p.C = sp.C;
      p.nblk = sp.nblk;
      p.out_cr = sp.out_cr;
      // X^T tiles: two boxes of 64 columns x 64 tokens
      if ((rc = make_map(&p.tmX, sp.X, sp.C, sp.T, sp.ldx, 64, 64)) != LORA_OK) return rc;
      int bytes = tile * 64 * 2;
      for (int k = 0; k < sp.nblk; ++k) {
        p.rs[k] = sp.rs[k];
        p.out[k] = sp.out[k];
        const int r8 = rank_pad8(sp.rs[k]);
        // S_b^T [rs_b, T]: 64 tokens x r8 rows, rows past rs_b zero-filled
        if ((rc = make_map(&p.tmS[k], sp.S[k], sp.T, sp.rs[k], sp.lds[k], 64, r8)) != LORA_OK) return rc;
        bytes += 64 * r8 * 2;
      }
      p.tx_bytes = bytes;
      p.rpad = rank_pad16(used_rank(sp.rs, sp.nblk));
      rmax = std::max(rmax, p.rpad);
      const int tiles = cdiv(p.C, tile);
      p.upt = cdiv(cdiv(p.T, 64), b.unit_chunks);
      p.unit_begin = b.units;
      b.units += tiles * p.upt;
      p.part_off = (long long)pf;
      p.red_begin = b.red_total;
      if (p.upt > 1) {
        pf += (size_t)tiles * p.upt * tile * p.rpad;
        b.red_total += tiles * tile * p.rpad;
      }
    }
    if (pf > ar.n_partials) return LORA_EWORKSPACE;  // planning bound violated
    b.partials = ar.partials;
    b.status = d->status;
    b.limit_ns = g_wait_limit_ns;
    if (launch_colmma(b, rmax, ctas, st) != cudaSuccess) return LORA_ECUDA;
  }
  return LORA_OK;
}

// ------------------------------------------------------------------ fused pass over dy
// sv = s dy B and dB = dy^T su of one projection in one read of dy.
struct DySpec {
  const bf* dy;
  int T, N, r;
  float scale;
  const bf* bt;   // B^T [pad8(r), N]
  const bf* sut;  // su^T [pad8(r), T]
  bf* sv;         // [T, pad8(r)]
  bf* svT;        // [pad8(r), T]
  float* dB;      // [N, r]
};

struct DyCut {
  int tt, groups, bpu, pieces;
};

constexpr int kDyTile = 128;  // tokens per tile and columns per block of the fused pass

size_t dy_sv_floats(int T, int rpad, int pieces) { return pieces > 1 ? (size_t)pieces * T * rpad : 0; }
size_t dy_db_floats(int N, int rpad, int groups) { return groups > 1 ? (size_t)groups * N * rpad : 0; }

// Token groups TMEM forces on a projection: each holds at most tiles_max tiles.
int dy_need_groups(int T, int tiles_max) { return cdiv(cdiv(T, kDyTile), tiles_max); }

// A projection takes the fused pass up to r = 16: beyond, the B^T and su^T
// boxes every stage carries (4 x 64 x r bf16 beside 32 KB of dy) make the one
// issuing thread's copies the limit, and the two separate passes are faster
// (Llama-3.2-3B layer, T = 2048, r = 32: 773 against 569 us; Qwen-2.5-3B
// layer, T = 4096, r = 64: 1254 against 944 us).  It also needs the partials
// of its fewest token groups to stay within a quarter of its dy bytes.
bool dy_fusable(int T, int N, int r) {
  const int rpad = rank_pad16(r);
  return rpad <= 16 && dy_db_floats(N, rpad, dy_need_groups(T, dy_tiles_max(rpad))) * 4 <= (size_t)T * N * 2 / 4;
}

// The cut of a projection for (gmul, pmul): gmul x the necessary token groups
// and pmul column pieces, trimmed (pieces first) until the partials fit within
// those of the necessary groups plus an eighth of the projection's dy bytes,
// or kDyPartialFloor floats for a small projection (whose few units would
// otherwise leave the side stream's SMs idle; 4 MB of partials cost ~1 us).
constexpr size_t kDyPartialFloor = size_t(1) << 20;
DyCut dy_cut(int T, int N, int rpad, int tiles_max, int gmul, int pmul) {
  const int tiles = cdiv(T, kDyTile), blocks = cdiv(N, kDyTile);
  const int need = dy_need_groups(T, tiles_max);
  int groups = std::min(tiles, std::min(need * gmul, std::max(need, kDyMaxCut)));
  int pieces = std::min(blocks, std::min(pmul, kDyMaxCut));
  const size_t cap = dy_db_floats(N, rpad, need) + std::max((size_t)T * N / 16, kDyPartialFloor);
  while (pieces > 1 && dy_sv_floats(T, rpad, pieces) + dy_db_floats(N, rpad, groups) > cap) --pieces;
  while (groups > need && dy_sv_floats(T, rpad, pieces) + dy_db_floats(N, rpad, groups) > cap) --groups;
  DyCut c;
  c.tt = cdiv(tiles, groups);
  c.groups = cdiv(tiles, c.tt);
  c.bpu = cdiv(blocks, pieces);
  c.pieces = cdiv(blocks, c.bpu);
  return c;
}

size_t dy_cut_floats(const DySpec& s, const DyCut& c) {
  const int rpad = rank_pad16(s.r);
  return dy_sv_floats(s.T, rpad, c.pieces) + dy_db_floats(s.N, rpad, c.groups);
}

// Cost of a batch's cuts on `ctas` persistent CTAs, in stage times (one
// 128 x 128 tile of dy): the units go round-robin in unit order, each costs its
// stages plus a fixed fill and its read-outs; partials add their traffic and
// the reduce launch.
double dy_cost(const std::vector<DySpec>& specs, size_t i0, size_t i1, const std::vector<DyCut>& cuts, int ctas) {
  std::vector<double> load(ctas, 0.0);
  long long u = 0;
  double part = 0.0;
  for (size_t i = i0; i < i1; ++i) {
    const DySpec& s = specs[i];
    const DyCut& c = cuts[i - i0];
    const int tiles = cdiv(s.T, kDyTile), blocks = cdiv(s.N, kDyTile), rpad = rank_pad16(s.r);
    for (int g = 0; g < c.groups; ++g) {
      const int nt = std::min(tiles, (g + 1) * c.tt) - g * c.tt;
      for (int q = 0; q < c.pieces; ++q, ++u) {
        const int nb = std::min(blocks, (q + 1) * c.bpu) - q * c.bpu;
        load[u % ctas] += nb * nt + 2.0 + nt * rpad / 64.0 + nb * rpad / 64.0;
      }
    }
    part += (double)dy_cut_floats(s, c);
  }
  const double make = *std::max_element(load.begin(), load.end());
  return part > 0 ? make + 4.0 + part * 8.0 / 32768.0 / ctas : make;
}

// The cuts of a batch (rank class of its largest rank) that cost least on
// `ctas` CTAs.  Choices are cached per shape set.
std::vector<DyCut> dy_choose(const std::vector<DySpec>& specs, size_t i0, size_t i1, int ctas) {
  static std::mutex mu;
  static std::map<std::vector<long long>, std::vector<DyCut>> cache;
  std::vector<long long> key{ctas};
  for (size_t i = i0; i < i1; ++i) key.insert(key.end(), {specs[i].T, specs[i].N, specs[i].r});
  {
    std::lock_guard<std::mutex> lk(mu);
    auto it = cache.find(key);
    if (it != cache.end()) return it->second;
  }
  int rmax = 16;
  for (size_t i = i0; i < i1; ++i) rmax = std::max(rmax, rank_pad16(specs[i].r));
  const int tmax = dy_tiles_max(rmax);
  std::vector<DyCut> best, cur(i1 - i0);
  double best_cost = 0.0;
  for (int gmul : {1, 2, 4, 8})
    for (int pmul : {1, 2, 4, 8}) {
      for (size_t i = i0; i < i1; ++i) cur[i - i0] = dy_cut(specs[i].T, specs[i].N, rank_pad16(specs[i].r), tmax, gmul, pmul);
      const double c = dy_cost(specs, i0, i1, cur, ctas);
      if (best.empty() || c < best_cost - 1e-9) {
        best = cur;
        best_cost = c;
      }
    }
  std::lock_guard<std::mutex> lk(mu);
  if (cache.size() > 4096) cache.clear();
  cache.emplace(key, best);
  return best;
}

// Partial floats a batch may need whatever the CTA count (the largest over every candidate cut).
size_t dy_worst_floats(const std::vector<DySpec>& specs, size_t i0, size_t i1) {
  int rmax = 16;
  for (size_t i = i0; i < i1; ++i) rmax = std::max(rmax, rank_pad16(specs[i].r));
  const int tmax = dy_tiles_max(rmax);
  size_t worst = 0;
  for (int gmul : {1, 2, 4, 8})
    for (int pmul : {1, 2, 4, 8}) {
      size_t f = 0;
      for (size_t i = i0; i < i1; ++i)
        f += dy_cut_floats(specs[i], dy_cut(specs[i].T, specs[i].N, rank_pad16(specs[i].r), tmax, gmul, pmul));
      worst = std::max(worst, f);
    }
  return worst;
}

size_t dy_plan_floats(const std::vector<DySpec>& specs) {
  size_t f = 0;
  for (size_t i0 = 0; i0 < specs.size(); i0 += kMaxRankProblems)
    f += dy_worst_floats(specs, i0, std::min(specs.size(), i0 + kMaxRankProblems));
  return f;
}

// The fused passes over dy on `ctas` persistent CTAs (one per SM), then their reduce; the cuts are
// the cheapest ones for `plan_ctas` CTAs (the cut decides how sv and dB are summed).
int launch_dy_pass(const std::vector<DySpec>& specs, const Arena& ar, const DeviceInfo* d, int ctas, int plan_ctas,
                   cudaStream_t st) {
  size_t pf = 0;
  int rc;
  for (size_t i0 = 0; i0 < specs.size(); i0 += kMaxRankProblems) {
    const size_t i1 = std::min(specs.size(), i0 + kMaxRankProblems);
    const std::vector<DyCut> cuts = dy_choose(specs, i0, i1, plan_ctas);
    DyBatch b;
    memset(&b, 0, sizeof(b));
    for (size_t i = i0; i < i1; ++i) {
      const DySpec& s = specs[i];
      const DyCut& c = cuts[i - i0];
      DyProb& p = b.p[b.n++];
      const int r8 = rank_pad8(s.r);
      if ((rc = make_map(&p.tmDy, s.dy, s.N, s.T, s.N, 64, kDyTile)) != LORA_OK) return rc;
      if ((rc = make_map(&p.tmBt, s.bt, s.N, s.r, s.N, 64, r8)) != LORA_OK) return rc;
      if ((rc = make_map(&p.tmSuT, s.sut, s.T, s.r, s.T, 64, r8)) != LORA_OK) return rc;
      p.T = s.T;
      p.N = s.N;
      p.r = s.r;
      p.rpad = rank_pad16(s.r);
      p.scale = s.scale;
      p.sv = s.sv;
      p.ld_sv = r8;
      p.svT = s.svT;
      p.dB = s.dB;
      p.tiles = cdiv(s.T, kDyTile);
      p.tt = c.tt;
      p.groups = c.groups;
      p.blocks = cdiv(s.N, kDyTile);
      p.bpu = c.bpu;
      p.pieces = c.pieces;
      p.unit_begin = b.units;
      b.units += c.groups * c.pieces;
      if (c.pieces > 1) {
        p.sv_part = (long long)pf;
        pf += dy_sv_floats(s.T, p.rpad, c.pieces);
        b.red_sv += s.T * (r8 / 8);
      }
      if (c.groups > 1) {
        p.db_part = (long long)pf;
        pf += dy_db_floats(s.N, p.rpad, c.groups);
        b.red_db += s.N * ((s.r + 3) / 4);
      }
    }
    if (pf > ar.n_partials) return LORA_EWORKSPACE;  // planning bound violated
    b.partials = ar.partials;
    b.status = d->status;
    b.limit_ns = g_wait_limit_ns;
    if (launch_dy(b, ctas, st) != cudaSuccess) return LORA_ECUDA;
  }
  return LORA_OK;
}

Arena arena(void* ws, const Plan& pl, int phase) {
  return Arena{at<float>(ws, pl.part_off[phase]), pl.n_partials[phase]};
}

// ------------------------------------------------------------------ forward
int add_fwd_problem(GemmBatch& b, const lora_proj& p, const Operands& o) {
  const lora_shape& s = p.shape;
  const int i = b.num_problems;
  const int64_t T = s.T, K = s.d_in, N = s.d_out, r = s.rank;
  int rc;
  // activation boxes: one CTA's 128 rows x 64 contraction elements; weight
  // boxes: 64 rows x 64 (two per CTA)
  if ((rc = make_map(&b.tmA[i], p.x, K, T, K, 64, 128)) != LORA_OK) return rc;
  // rank 0: no adapter slab (kb_total = kb_main), so the slab maps are never read
  if ((rc = r > 0 ? make_map(&b.tmA2[i], o.s_in, r, T, o.ld_s, 64, 128) : (b.tmA2[i] = b.tmA[i], LORA_OK)) != LORA_OK)
    return rc;
  if (is_q4(p)) {
    // 4-bit W: a box is 64 rows x 64 codes (32 bytes); (s, b) boxes are 128 rows x 4 groups
    if ((rc = make_map_plain(&b.tmQ[i], CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, p.Wq.codes, K / 2, N, K / 2, 32, 64)) !=
        LORA_OK)
      return rc;
    if ((rc = make_map_plain(&b.tmP[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, p.Wq.params, K / 32, N, K / 32, 8,
                             128)) != LORA_OK)
      return rc;
  } else if ((rc = make_map(&b.tmB[i], p.W, K, N, K, 64, 64)) != LORA_OK) {
    return rc;
  }
  if ((rc = r > 0 ? make_map(&b.tmB2[i], o.B, r, N, o.ld_b, 64, 64) : (b.tmB2[i] = b.tmA[i], LORA_OK)) != LORA_OK)
    return rc;
  if ((rc = make_map(&b.tmOut[i], p.y, N, T, N, 64, 32)) != LORA_OK) return rc;
  GemmProblem& g = b.prob[i];
  gemm_shape(g, T, N, K, r);
  g.out = mb(p.y);
  add_problem(b);
  return LORA_OK;
}

// ------------------------------------------------------------------ backward
int add_bwd_problem(GemmBatch& b, const lora_proj& p, const Operands& o) {
  const lora_shape& s = p.shape;
  const int i = b.num_problems;
  const int64_t T = s.T, K = s.d_in, N = s.d_out, r = s.rank;
  int rc;
  if ((rc = make_map(&b.tmA[i], p.dy, N, T, N, 64, 128)) != LORA_OK) return rc;
  if ((rc = r > 0 ? make_map(&b.tmA2[i], o.s_in, r, T, o.ld_s, 64, 128) : (b.tmA2[i] = b.tmA[i], LORA_OK)) != LORA_OK)
    return rc;
  // W [N, K] read MN-major: inner dimension K (the GEMM's output columns), rows = contraction
  if (is_q4(p)) {
    // 4-bit W: a box is 64 rows x 128 codes (64 bytes); (s, b) boxes are 64 rows x 4 groups
    if ((rc = make_map_plain(&b.tmQ[i], CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, p.Wq.codes, K / 2, N, K / 2, 64, 64)) !=
        LORA_OK)
      return rc;
    if ((rc = make_map_plain(&b.tmP[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, p.Wq.params, K / 32, N, K / 32, 8,
                             64)) != LORA_OK)
      return rc;
  } else if ((rc = make_map(&b.tmB[i], p.W, K, N, K, 64, 64)) != LORA_OK) {
    return rc;
  }
  if ((rc = r > 0 ? make_map(&b.tmB2[i], p.A, K, r, K, 64, 64) : (b.tmB2[i] = b.tmA[i], LORA_OK)) != LORA_OK)
    return rc;
  if ((rc = make_map(&b.tmOut[i], p.dx, K, T, K, 64, 32)) != LORA_OK) return rc;
  GemmProblem& g = b.prob[i];
  gemm_shape(g, T, K, N, r);
  g.out = mb(p.dx);
  add_problem(b);
  return LORA_OK;
}

void init_batch(GemmBatch& b, const DeviceInfo* d) {
  memset(&b, 0, sizeof(b));
  b.status = d->status;
  b.limit_ns = g_wait_limit_ns;
}

// ------------------------------------------------------------------ checks
// The base weight: bf16 W, or 4-bit codes with their (s, b) pairs (exactly one).
int check_weight(const lora_proj& p) {
  const bool q = p.Wq.codes != nullptr || p.Wq.params != nullptr;
  if (q && p.W) return LORA_EINVAL;
  if (!q) return p.W ? LORA_OK : LORA_ENULL;
  if (!p.Wq.codes || !p.Wq.params) return LORA_ENULL;
  if (p.shape.d_in % 256) return LORA_EINVAL;  // whole 64-wide groups, 16-byte (s, b) rows
  if (!aligned16(p.Wq.codes) || !aligned16(p.Wq.params)) return LORA_EALIGN;
  return LORA_OK;
}

// A frozen projection (rank 0) has no adapter: A, B, su, dA and dB are neither read nor written.
int check_fwd_ptrs(const lora_proj& p) {
  if (!p.x || !p.y) return LORA_ENULL;
  if (p.shape.rank > 0 && (!p.A || !p.B)) return LORA_ENULL;
  const void* ps[] = {p.x, p.W, p.A, p.B, p.y, p.su};
  for (const void* q : ps)
    if (q && !aligned16(q)) return LORA_EALIGN;
  return check_weight(p);
}

int check_bwd_ptrs(const lora_proj& p) {
  if (!p.dy || !p.x) return LORA_ENULL;
  if (p.shape.rank > 0 && (!p.A || !p.B || !p.su || !p.dA || !p.dB)) return LORA_ENULL;
  const void* ps[] = {p.dy, p.x, p.W, p.A, p.B, p.su, p.dx, p.dA, p.dB};
  for (const void* q : ps)
    if (q && !aligned16(q)) return LORA_EALIGN;
  return check_weight(p);
}

int check_ws(void* ws, size_t ws_bytes, size_t need) {
  if (!ws || ws_bytes < need) return LORA_EWORKSPACE;
  if (reinterpret_cast<uintptr_t>(ws) & 255u) return LORA_EALIGN;
  return LORA_OK;
}

// Side-stream schedule of a forward-and-backward call: fork after the
// forward's row products; the dx contraction waits for sv, the end of the call
// for dA and dB.  Each host thread has its own side stream and events per
// device, so a stream capture on one thread never takes in another thread's
// work; they are created on a thread's first such call and kept.
bool overlap_enabled() {
  static const bool on = [] {
    const char* e = getenv("LORA_OVERLAP");
    return !(e && e[0] == '0' && e[1] == 0);
  }();
  return on;
}

// Widths of the side stream in its two phases.  Beside the forward
// contraction (2TKN FLOPs per projection, compute-bound, 4-bit weights ~1.3x
// slower per FLOP) it transposes B and su and reads dy once: the fused pass
// (sv and dB, r <= 16) or the sv pass; the dx contraction waits for sv.
// Beside the dx contraction it runs dA = sv^T x (2TK bytes per distinct x) and,
// where the pass over dy was not fused, dB (dy read again, 0.6 x as costly
// per byte).  The rank-r kernels are issue-bound, costlier per byte as r
// grows.  Each phase gets the share of SMs that ends it with the contraction
// beside it:
//   w / (SMs - w) = kappa x side bytes of the phase / contraction FLOPs,
// side bytes = 2T(...)(1 + r / 144) + an adapter-sized term (transposes,
// partial sums, fp32 gradients).  kappa1 gives the Llama-3.2-3B layer at
// r = 16 12 SMs, kappa2 8 SMs, the measured best pair at T = 2048; the same
// constants give 16 / 8 for the Qwen-2.5-3B layer at r = 16 (best measured
// 16-18 / 8) and 22 / 20 at r = 64 (best 16-20 / 20-24).  Rounded to even
// counts so the contractions keep whole CTA pairs; LORA_SIDE_SMS and
// LORA_SIDE_SMS2 override.
constexpr double kSideKappa1 = 290.0;
constexpr double kSideKappa2 = 245.0;
constexpr double kSideAdapter1 = 12.0;  // bytes per r N
constexpr double kSideAdapter2 = 8.0;   // bytes per r K
constexpr double kSideSecondPass = 0.6;  // the unfused dB pass over dy: its kernel streams faster per byte

struct SideWidths {
  int w1 = 0, w2 = 0;
};

int env_int(const char* name) {
  const char* e = getenv(name);
  return e ? atoi(e) : 0;
}

bool dy_fusable(int T, int N, int r);

SideWidths side_widths(int num_sms, const lora_proj* projs, int n) {
  static const int v1 = env_int("LORA_SIDE_SMS"), v2 = env_int("LORA_SIDE_SMS2");
  double b1 = 0.0, b2 = 0.0, flops = 0.0;
  std::vector<const void*> xs;
  for (int i = 0; i < n; ++i) {
    const lora_shape& sh = projs[i].shape;
    const double T = (double)sh.T, K = (double)sh.d_in, N = (double)sh.d_out, r = (double)sh.rank;
    flops += 2.0 * T * K * N * (is_q4(projs[i]) ? 1.3 : 1.0);
    if (sh.rank == 0) continue;  // a frozen projection puts no work on the side stream
    const double fr = 1.0 + r / 144.0;
    b1 += 2.0 * T * N * fr + kSideAdapter1 * r * N;
    b2 += kSideAdapter2 * r * K;
    if (!dy_fusable((int)sh.T, (int)sh.d_out, (int)sh.rank)) b2 += kSideSecondPass * 2.0 * T * N * fr;
    // dA reads each distinct x once (shapes without pointers: once per projection)
    const void* x = projs[i].x;
    if (x == nullptr || std::find(xs.begin(), xs.end(), x) == xs.end()) {
      b2 += 2.0 * T * K * fr;
      if (x != nullptr) xs.push_back(x);
    }
  }
  auto width = [&](double kappa, double bytes) {
    const double c = flops > 0.0 ? kappa * bytes / flops : 0.0;
    return 2 * (int)std::lround(num_sms * c / (1.0 + c) / 2.0);
  };
  SideWidths w;
  w.w1 = std::max(2, std::min(num_sms / 4, v1 > 0 ? v1 : width(kSideKappa1, b1)));
  w.w2 = std::max(2, std::min(num_sms / 4, v2 > 0 ? v2 : width(kSideKappa2, b2)));
  // A contraction with few output tiles runs as a cluster split, four CTAs per 256 x 256 tile, and leaves
  // the other SMs idle: the side stream takes them (the split still fits beside it).
  auto cs_sms = [&](bool bwd, int side) {
    long long wide = 0, narrow = 0;
    for (int i = 0; i < n; ++i) {
      if (is_q4(projs[i])) return 0;  // 4-bit weights keep the wide tiles
      const lora_shape& sh = projs[i].shape;
      const int out = bwd ? sh.d_in : sh.d_out, depth = bwd ? sh.d_out : sh.d_in;
      const int kb = cdiv(depth, 64) + (sh.rank > 0 ? cdiv(sh.rank, 64) : 0);
      if (kb < kCsMinBlocks || kb > kCsMaxBlocks) return 0;
      wide += (long long)cdiv(sh.T, 256) * cdiv(out, gemm_tile_n());
      narrow += (long long)cdiv(sh.T, 256) * cdiv(out, gemm_tile_n_f32());
    }
    const int pairs = (num_sms - side) / 2;
    if (wide == 0 || wide >= pairs || 2 * narrow > pairs || narrow > gemm_cs_max_clusters(bwd)) return 0;
    return (int)(4 * narrow);
  };
  if (v1 <= 0) {
    const int used = cs_sms(false, w.w1);
    if (used > 0) w.w1 = std::max(w.w1, (num_sms - used) & ~1);
  }
  if (v2 <= 0) {
    const int used = cs_sms(true, w.w2);
    if (used > 0) w.w2 = std::max(w.w2, (num_sms - used) & ~1);
  }
  return w;
}

// Whether any projection has an adapter (rank > 0): frozen ones have no rank-r work.
bool any_adapter(const lora_proj* projs, int n) {
  for (int i = 0; i < n; ++i)
    if (projs[i].shape.rank > 0) return true;
  return false;
}

struct SideCtx {
  cudaStream_t side = nullptr;
  cudaEvent_t ev[3] = {nullptr, nullptr, nullptr};  // fork, sv ready, side done
};

struct ThreadSide {
  SideCtx dev[kMaxDevices];
  ~ThreadSide() {
    for (SideCtx& c : dev) {
      for (cudaEvent_t e : c.ev)
        if (e) cudaEventDestroy(e);
      if (c.side) cudaStreamDestroy(c.side);
    }
  }
};

thread_local ThreadSide t_side;

struct Overlap {
  bool on = false, forked = false, joined = false;
  int side_ctas = 0;   // beside the forward contraction
  int side_ctas2 = 0;  // beside the dx contraction
  cudaStream_t main = nullptr, side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_sv = nullptr, ev_done = nullptr;
  int init(const DeviceInfo* d, cudaStream_t st, const lora_proj* projs, int n) {
    if (!overlap_enabled() || !any_adapter(projs, n)) return LORA_OK;
    SideCtx& c = t_side.dev[d - g_dev];
    if (!c.side && cudaStreamCreateWithFlags(&c.side, cudaStreamNonBlocking) != cudaSuccess) return LORA_ECUDA;
    for (cudaEvent_t& e : c.ev)
      if (!e && cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess) return LORA_ECUDA;
    main = st;
    side = c.side;
    ev_fork = c.ev[0];
    ev_sv = c.ev[1];
    ev_done = c.ev[2];
    const SideWidths w = side_widths(d->num_sms, projs, n);
    side_ctas = w.w1;
    side_ctas2 = w.w2;
    on = true;
    return LORA_OK;
  }
  int fork() {
    forked = true;
    return cudaEventRecord(ev_fork, main) == cudaSuccess && cudaStreamWaitEvent(side, ev_fork, 0) == cudaSuccess
               ? LORA_OK
               : LORA_ECUDA;
  }
  int wait_sv() { return cudaStreamWaitEvent(main, ev_sv, 0) == cudaSuccess ? LORA_OK : LORA_ECUDA; }
  // the call ends when everything it put on the side stream is done
  int join() {
    joined = true;
    return cudaEventRecord(ev_done, side) == cudaSuccess && cudaStreamWaitEvent(main, ev_done, 0) == cudaSuccess
               ? LORA_OK
               : LORA_ECUDA;
  }
  ~Overlap() {
    if (forked && !joined) join();  // an error after the fork: still end after the side work
  }
};

// Runs the given projections in `mode`; every argument already validated.
int run_step(const lora_proj* projs, int n, int mode, void* ws, const Plan& pl, DeviceInfo* d, cudaStream_t st) {
  int rc;
  const std::vector<Ws>& plans = pl.ws;
  auto W_ = [&](int i) { return at<uint8_t>(ws, pl.offs[i]); };
  // tile counters of the fused-GEMM launches
  int* counters = at<int>(ws, 0);
  int next_counter = 0;
  if (cudaMemsetAsync(ws, 0, pl.zero_bytes, st) != cudaSuccess) return LORA_ECUDA;
  // whether a kernel of this call already ran on the main stream: a contraction launched after one may
  // load its base operands (inputs of the call) before the previous grid ends
  bool prior_main = false;
  // forward and backward in one call: the backward's rank-r work runs on a side
  // stream with a few SMs while the contractions use the rest; a backward alone
  // computes sv (which the dx contraction reads) first on every SM, then dA (and
  // dB where the pass over dy is not fused) on the side stream beside the dx
  // contraction
  Overlap ov;
  if ((mode & LORA_BWD) && (rc = ov.init(d, st, projs, n)) != LORA_OK) return rc;
  const int gemm_sms = ov.on ? d->num_sms - ov.side_ctas : d->num_sms;      // forward contraction
  const int gemm_sms_b = ov.on ? d->num_sms - ov.side_ctas2 : d->num_sms;  // dx contraction
  // backward rank-r work: B^T, su^T, sv (and sv^T), then dB and dA; on `rs`
  // with `ctas` persistent CTAs; the operands of the dx contraction go to bops
  std::vector<Operands> bops(n);
  // ctas: CTAs of the transposes and the passes over dy, on rs; ctas2: of dA (and
  // the second pass over dy where it is not fused), on rs2 (after rs's first phase)
  auto bwd_rank = [&](cudaStream_t rs, int ctas, cudaStream_t rs2, int ctas2) -> int {
    int rc;
    std::vector<RowSpec> rows;
    std::vector<ColSpec> cols;
    std::vector<DySpec> dys;
    std::vector<bf*> sut(n), svt(n);
    std::vector<char> fused(n);
    for (int i = 0; i < n; ++i)
      fused[i] = projs[i].shape.rank > 0 &&
                 dy_fusable((int)projs[i].shape.T, (int)projs[i].shape.d_out, (int)projs[i].shape.rank);
    std::vector<Operands>& ops = bops;
    TransposeJobs tj;
    memset(&tj, 0, sizeof(tj));
    {
      ProfScope ps(LORA_KERNEL_PAD, rs);
      // rank sides as K-major tensor-core operands: B^T for sv = s dy B and
      // su^T for dB = dy^T su, zero rows past r
      auto transpose = [&](const bf* src, int rows_, int r, bf* dst) -> int {
        if (tj.count == kMaxTransposes) {
          if (launch_transposes(tj, rs) != cudaSuccess) return LORA_ECUDA;
          memset(&tj, 0, sizeof(tj));
        }
        const int k = tj.count++;
        tj.src[k] = src;
        tj.dst[k] = dst;
        tj.n[k] = rows_;
        tj.r[k] = r;
        tj.ld[k] = r;
        tj.r8[k] = rank_pad8(r);
        tj.max_elems = std::max(tj.max_elems, (long long)rows_ * tj.r8[k]);
        return LORA_OK;
      };
      for (int i = 0; i < n; ++i) {
        const lora_proj& p = projs[i];
        const int T = (int)p.shape.T, N = (int)p.shape.d_out, r = (int)p.shape.rank, r8 = rank_pad8(r);
        if (r == 0) continue;  // frozen: dx = dy W only
        bf* bt = at<bf>(W_(i), plans[i].bt);
        sut[i] = at<bf>(W_(i), plans[i].sut);
        svt[i] = at<bf>(W_(i), plans[i].svt);
        if ((rc = transpose(cb(p.B), N, r, bt)) != LORA_OK) return rc;
        if ((rc = transpose(cb(p.su), T, r, sut[i])) != LORA_OK) return rc;
        bf* sv = at<bf>(W_(i), plans[i].sv);
        if (fused[i])
          dys.push_back(DySpec{cb(p.dy), T, N, r, p.shape.scale, bt, sut[i], sv, svt[i], p.dB});
        else
          add_row_block(rows, cb(p.dy), N, T, N, p.shape.scale, bt, N, r, sv, r8, nullptr, 0, svt[i], false);
        ops[i].s_in = sv;
        ops[i].ld_s = r8;
      }
      if (launch_transposes(tj, rs) != cudaSuccess) return LORA_ECUDA;
    }
    {
      // sv (and dB where fused) before the event the dx contraction waits for
      ProfScope ps(LORA_KERNEL_ROWPROJ, rs);
      if ((rc = launch_dy_pass(dys, arena(ws, pl, kPhBwdRows), d, ctas, pl.dy_cut_device ? d->num_sms : ctas, rs)) !=
          LORA_OK)
        return rc;
      if ((rc = launch_rows(rows, arena(ws, pl, kPhBwdRows), d, ctas, rs)) != LORA_OK) return rc;
    }
    // sv is complete: the dx contraction may start (on the main stream: at once, or after this event)
    if (ov.on && rs != ov.main && cudaEventRecord(ov.ev_sv, rs) != cudaSuccess) return LORA_ECUDA;
    if (ov.on && rs == ov.main && rs2 != rs && (rc = ov.fork()) != LORA_OK) return rc;
    for (int i = 0; i < n; ++i) {
      if (fused[i] || projs[i].shape.rank == 0) continue;
      const lora_proj& p = projs[i];
      const int T = (int)p.shape.T, N = (int)p.shape.d_out, r = (int)p.shape.rank;
      add_col_block(cols, cb(p.dy), N, T, N, sut[i], T, r, p.dB, 1, false);
    }
    for (int i = 0; i < n; ++i) {
      const lora_proj& p = projs[i];
      const int T = (int)p.shape.T, K = (int)p.shape.d_in, r = (int)p.shape.rank;
      if (r > 0) add_col_block(cols, cb(p.x), K, T, K, svt[i], T, r, p.dA, 0, true);
    }
    {
      ProfScope ps(LORA_KERNEL_COLPROJ, rs2);
      if ((rc = launch_cols(cols, arena(ws, pl, kPhBwdCols), d, ctas2, rs2)) != LORA_OK) return rc;
    }
    return LORA_OK;
  };
  if (mode & LORA_FWD) {
    std::vector<Operands> ops(n);
    std::vector<RowSpec> rows;
    {
      ProfScope ps(LORA_KERNEL_PAD, st);
      for (int i = 0; i < n; ++i) {
        const lora_proj& p = projs[i];
        const int T = (int)p.shape.T, K = (int)p.shape.d_in, N = (int)p.shape.d_out, r = (int)p.shape.rank;
        const int r8 = rank_pad8(r);
        const bool pad = (r % 8) != 0;
        if (r == 0) continue;  // frozen: y = x W^T only
        bf* su_gemm = (p.su && !pad) ? mb(p.su) : at<bf>(W_(i), plans[i].su_pad);
        const int ld_gemm = (p.su && !pad) ? r : r8;
        bf* su_user2 = (p.su && pad) ? mb(p.su) : nullptr;
        add_row_block(rows, cb(p.x), K, T, K, p.shape.scale, cb(p.A), K, r, su_gemm, ld_gemm, su_user2, r, nullptr,
                      true);
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
      if ((rc = launch_rows(rows, arena(ws, pl, kPhFwdRows), d, d->num_sms, st)) != LORA_OK) return rc;
    }
    if (!rows.empty()) prior_main = true;
    // the backward's rank-r work needs su only: it may start now, beside the forward contractions
    if (ov.on && (rc = ov.fork()) != LORA_OK) return rc;
    if (ov.on && (rc = bwd_rank(ov.side, ov.side_ctas, ov.side, ov.side_ctas2)) != LORA_OK) return rc;
    // one launch per batch of bf16-weight, then of 4-bit-weight problems;
    // heavier problems first so that the tile walk ends balanced
    for (int q4 = 0; q4 < 2; ++q4) {
      std::vector<int> order;
      for (int i = 0; i < n; ++i)
        if (is_q4(projs[i]) == (q4 != 0)) order.push_back(i);
      std::stable_sort(order.begin(), order.end(),
                       [&](int a, int b) { return projs[a].shape.d_in > projs[b].shape.d_in; });
      for (size_t i0 = 0; i0 < order.size(); i0 += kMaxProblems) {
        GemmBatch b;
        init_batch(b, d);
        b.tile_counter = counters + next_counter++;
        b.early_inputs = prior_main ? 1 : 0;
        prior_main = true;
        int sp[kMaxProblems];
        float* parts[kMaxProblems];
        for (size_t i = i0; i < order.size() && i < i0 + kMaxProblems; ++i) {
          if ((rc = add_fwd_problem(b, projs[order[i]], ops[order[i]])) != LORA_OK) return rc;
          sp[i - i0] = pl.split_f[order[i]];
          parts[i - i0] = at<float>(ws, pl.split_off[order[i]]);
        }
        ProfScope ps(LORA_KERNEL_GEMM_FWD, st);
        if (q4 == 0 && use_cluster_split(b, false, gemm_sms / 2)) {
          if (launch_fused_gemm_cs(b, false, st) != cudaSuccess) return LORA_ECUDA;
          continue;
        }
        if ((rc = apply_splits(b, sp, parts)) != LORA_OK) return rc;
        if (launch_fused_gemm(b, false, q4 != 0, gemm_sms, st) != cudaSuccess) return LORA_ECUDA;
        if (launch_split_reduce(b, st) != cudaSuccess) return LORA_ECUDA;
      }
    }
  }
  if (mode & LORA_BWD) {
    // (a forward-and-backward call without the side stream runs it here too, on every SM)
    if (!(mode == LORA_FWD_BWD && ov.on)) {
      if ((rc = bwd_rank(st, d->num_sms, ov.on ? ov.side : st, ov.on ? ov.side_ctas2 : d->num_sms)) != LORA_OK)
        return rc;
      if (any_adapter(projs, n)) prior_main = true;  // the pass over dy or the row products ran here
    }
    // the dx contraction reads sv: when the side stream computed it, wait for it
    if (mode == LORA_FWD_BWD && ov.on && (rc = ov.wait_sv()) != LORA_OK) return rc;
    std::vector<Operands>& ops = bops;
    for (int q4 = 0; q4 < 2; ++q4) {
      std::vector<int> order;
      for (int i = 0; i < n; ++i)
        if (projs[i].dx && is_q4(projs[i]) == (q4 != 0)) order.push_back(i);
      std::stable_sort(order.begin(), order.end(),
                       [&](int a, int b) { return projs[a].shape.d_out > projs[b].shape.d_out; });
      for (size_t i0 = 0; i0 < order.size(); i0 += kMaxProblems) {
        GemmBatch b;
        init_batch(b, d);
        b.tile_counter = counters + next_counter++;
        b.early_inputs = prior_main ? 1 : 0;
        prior_main = true;
        int sp[kMaxProblems];
        float* parts[kMaxProblems];
        for (size_t i = i0; i < order.size() && i < i0 + kMaxProblems; ++i) {
          if ((rc = add_bwd_problem(b, projs[order[i]], ops[order[i]])) != LORA_OK) return rc;
          sp[i - i0] = pl.split_b[order[i]];
          parts[i - i0] = at<float>(ws, pl.split_off[order[i]]);
        }
        ProfScope ps(LORA_KERNEL_GEMM_BWD, st);
        if (q4 == 0 && use_cluster_split(b, true, gemm_sms_b / 2)) {
          if (launch_fused_gemm_cs(b, true, st) != cudaSuccess) return LORA_ECUDA;
          continue;
        }
        if ((rc = apply_splits(b, sp, parts)) != LORA_OK) return rc;
        if (launch_fused_gemm(b, true, q4 != 0, gemm_sms_b, st) != cudaSuccess) return LORA_ECUDA;
        if (launch_split_reduce(b, st) != cudaSuccess) return LORA_ECUDA;
      }
    }
  }
  // the call ends when the side stream's dA and dB are done
  if (ov.on && (rc = ov.join()) != LORA_OK) return rc;
  return LORA_OK;
}

// allow_split false: every contraction in one pass (the fixed-scratch forward keeps its footprint).
int plan_all(const lora_proj* projs, int n, int mode, Plan* pl, bool allow_split = true) {
  // partials are bounded by the smallest unit size (most units per tile)
  const int tile = rank_mma_tile();
  auto upt = [&](int64_t len) { return (size_t)cdiv(cdiv(len, 64), kMinUnitChunks); };
  auto tiles = [&](int64_t len) { return (size_t)cdiv(len, tile); };
  std::vector<DySpec> dy_shapes;  // the fused passes over dy, in the order the backward forms them
  size_t rows_bwd = 0;
  for (int i = 0; i < n; ++i) {
    int rc = check_shape(&projs[i].shape);
    if (rc != LORA_OK) return rc;
    const lora_shape& s = projs[i].shape;
    const size_t r16 = (size_t)rank_pad16((int)s.rank);
    if (s.rank == 0) continue;  // frozen projection: no rank-r work
    if ((mode & LORA_FWD) && upt(s.d_in) > 1) pl->n_partials[kPhFwdRows] += tiles(s.T) * upt(s.d_in) * tile * r16;
    if (mode & LORA_BWD) {
      const bool fused = dy_fusable((int)s.T, (int)s.d_out, (int)s.rank);
      if (fused)
        dy_shapes.push_back(DySpec{nullptr, (int)s.T, (int)s.d_out, (int)s.rank, s.scale, nullptr, nullptr, nullptr,
                                   nullptr, nullptr});
      else if (upt(s.d_out) > 1)
        rows_bwd += tiles(s.T) * upt(s.d_out) * tile * r16;
      if (upt(s.T) > 1) pl->n_partials[kPhBwdCols] += ((fused ? 0 : tiles(s.d_out)) + tiles(s.d_in)) * upt(s.T) * tile * r16;
    }
  }
  // the fused passes over dy and the remaining row products run one after the other: one arena
  pl->n_partials[kPhBwdRows] = std::max(rows_bwd, dy_plan_floats(dy_shapes));
  // split contractions: batches as run_step forms them (every projection counted for the backward)
  pl->split_f.assign(n, 1);
  pl->split_b.assign(n, 1);
  // the side stream's SMs are left out of the contractions they run beside: the
  // forward's in a forward-and-backward call, the dx contraction's in any call with a backward
  int pairs_dir[2] = {kPlanPairs, kPlanPairs};
  // pair counts the partials are also sized for: every pair, and the side widths of the same shapes with
  // bf16 and with 4-bit weights, so that a size reported from the shapes alone (lora_workspace_size)
  // covers a call of either weight kind in any mode
  std::vector<int> pairs_alt[2] = {{kPlanPairs}, {kPlanPairs}};
  if ((mode & LORA_BWD) && overlap_enabled() && any_adapter(projs, n)) {
    const SideWidths w = side_widths(kPlanSms, projs, n);
    if (mode == LORA_FWD_BWD) pairs_dir[0] = (kPlanSms - w.w1) / 2;
    pairs_dir[1] = (kPlanSms - w.w2) / 2;
    static const uint8_t kAnyCodes = 0;  // a non-null code pointer marks a projection 4-bit for the widths
    for (int q4 = 0; q4 < 2; ++q4) {
      std::vector<lora_proj> as(projs, projs + n);
      for (lora_proj& p : as) p.Wq.codes = q4 ? &kAnyCodes : nullptr;
      const SideWidths wa = side_widths(kPlanSms, as.data(), n);
      pairs_alt[0].push_back((kPlanSms - wa.w1) / 2);
      pairs_alt[1].push_back((kPlanSms - wa.w2) / 2);
    }
  }
  std::vector<size_t> split_need(n, 0);
  for (int dir = 0; dir < 2; ++dir) {
    if (!(mode & (dir == 0 ? LORA_FWD : LORA_BWD))) continue;
    for (int q4 = 0; q4 < 2; ++q4) {
      std::vector<int> order;
      for (int i = 0; i < n; ++i)
        if (is_q4(projs[i]) == (q4 != 0)) order.push_back(i);
      std::stable_sort(order.begin(), order.end(), [&](int a, int b) {
        return dir == 0 ? projs[a].shape.d_in > projs[b].shape.d_in : projs[a].shape.d_out > projs[b].shape.d_out;
      });
      for (size_t i0 = 0; i0 < order.size(); i0 += kMaxProblems) {
        GemmBatch b;
        memset(&b, 0, sizeof(b));
        for (size_t i = i0; i < order.size() && i < i0 + kMaxProblems; ++i) {
          const lora_shape& sh = projs[order[i]].shape;
          if (dir == 0)
            gemm_shape(b.prob[b.num_problems], sh.T, sh.d_out, sh.d_in, sh.rank);
          else
            gemm_shape(b.prob[b.num_problems], sh.T, sh.d_in, sh.d_out, sh.rank);
          add_problem(b);
        }
        // the splits for the pairs this call's contraction gets, and the partials sized for the
        // largest of those splits and the ones for the other pair counts above: a forward-and-backward
        // call's workspace, whose side stream may leave few pairs to a contraction, must also hold a
        // forward or backward call of the same shapes
        for (size_t pass = 0; pass <= pairs_alt[dir].size(); ++pass) {
          const int pairs = pass == 0 ? pairs_dir[dir] : pairs_alt[dir][pass - 1];
          if (pass > 0 && pairs == pairs_dir[dir]) continue;
          int sp[kMaxProblems];
          choose_splits(b, sp, pairs);
          if (!allow_split)
            for (int q = 0; q < b.num_problems; ++q) sp[q] = 1;
          for (int q = 0; q < b.num_problems; ++q) {
            const int pi = order[i0 + q];
            if (pass == 0) (dir == 0 ? pl->split_f : pl->split_b)[pi] = sp[q];
            split_need[pi] = std::max(split_need[pi], split_floats(b.prob[q], sp[q]));
          }
        }
      }
    }
  }
  size_t off = kWsHeader;
  pl->zero_bytes = off;
  for (int k = 0; k < kPhases; ++k) {
    pl->part_off[k] = off;
    off += up256(pl->n_partials[k] * sizeof(float));
  }
  pl->split_off.assign(n, 0);
  for (int i = 0; i < n; ++i) {
    pl->split_off[i] = off;
    off += split_need[i] * sizeof(float);
  }
  pl->ws.resize(n);
  pl->offs.resize(n);
  for (int i = 0; i < n; ++i) {
    pl->ws[i] = plan_ws(projs[i].shape, mode);
    pl->offs[i] = off;
    off += up256(pl->ws[i].total);
  }
  pl->total = off;
  return LORA_OK;
}


// Checkpointed stack (Algorithm 2): scratch for one layer's saved su (the
// largest layer) and for one stack step.
int ckpt_layout(const lora_proj* projs, int n_layers, int n_per, size_t* su_bytes, size_t* step_bytes) {
  if (!projs) return LORA_ENULL;
  if (n_layers < 1 || n_per < 1 || n_per > 64) return LORA_EINVAL;
  size_t sb = 0, wb = 0;
  for (int l = 0; l < n_layers; ++l) {
    const lora_proj* L = projs + (size_t)l * n_per;
    size_t su = 0;
    for (int i = 0; i < n_per; ++i) {
      int rc = check_shape(&L[i].shape);
      if (rc != LORA_OK) return rc;
      su += up256((size_t)L[i].shape.T * (size_t)L[i].shape.rank * 2);
    }
    Plan pl;
    int rc = plan_all(L, n_per, LORA_FWD_BWD, &pl);  // bounds the su-less forward's needs too
    if (rc != LORA_OK) return rc;
    sb = std::max(sb, su);
    wb = std::max(wb, pl.total);
  }
  *su_bytes = up256(sb);
  *step_bytes = wb;
  return LORA_OK;
}

// One layer's projections with su placed in the scratch (or NULL).
void layer_copy(const lora_proj* L, int n_per, uint8_t* su_scratch, std::vector<lora_proj>* out) {
  out->assign(L, L + n_per);
  size_t off = 0;
  for (int i = 0; i < n_per; ++i) {
    (*out)[i].su = su_scratch ? reinterpret_cast<lora_bf16*>(su_scratch + off) : nullptr;
    off += up256((size_t)L[i].shape.T * (size_t)L[i].shape.rank * 2);
  }
}


// ------------------------------------------------------------------ reduced-vocabulary cross entropy

// Split partials of one contraction: splits happen only below kPlanPairs output
// tiles (M x N < kPlanPairs 256 x 512 padded), at most 8 of them.
constexpr size_t kCeSplitFloats = (size_t)8 * kPlanPairs * 256 * 512 + 64 * 1024;

struct CePlan {
  size_t flags, counts, segs, J, pos, tl, tpos, ycol, rowloss, lse, ht, ej, z, lse_part, g, dht, part, tiles, total;
  int ld_lse;
};

int ce_check(const lora_ce_args* a, CePlan* pl) {
  if (!a) return LORA_ENULL;
  if (a->T < 1 || a->V < 1 || a->d < 8 || (a->d % 8) || a->T > (1ll << 24) || a->V > (1ll << 24) ||
      a->d > (1ll << 20))
    return LORA_EINVAL;
  if (a->topk && (a->k < 1 || a->ld_topk < a->k)) return LORA_EINVAL;
  if (!a->h || !a->E || !a->targets || !a->loss) return LORA_ENULL;
  const void* ps[] = {a->h, a->E, a->dh};
  for (const void* q : ps)
    if (q && !aligned16(q)) return LORA_EALIGN;
  const int64_t T = a->T, V = a->V, d = a->d;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += up256(bytes);
    return o;
  };
  pl->tiles = take(16);
  pl->counts = take(32);  // |T_set|, |J|, error flag, -, two last-block counters
  pl->segs = take(128 * 4);
  pl->flags = take((size_t)V);
  pl->J = take((size_t)V * 4);
  pl->pos = take((size_t)V * 4);
  pl->tl = take((size_t)T * 4);
  pl->tpos = take((size_t)T * 4);
  pl->ycol = take((size_t)T * 4);
  pl->rowloss = take((size_t)T * 4);
  pl->lse = take((size_t)T * 4);
  pl->ht = take((size_t)T * d * 2);
  // J is the whole vocabulary without a top-k table: E is read in place
  pl->ej = take(a->topk ? (size_t)V * d * 2 : 0);
  pl->z = take((size_t)T * rup(V, 4) * 4);
  pl->ld_lse = (int)cdiv(V, gemm_lse_group());
  pl->lse_part = take((size_t)T * pl->ld_lse * 8);
  pl->g = take((size_t)T * rup(V, 8) * 2);
  pl->dht = take((size_t)T * d * 2);
  pl->part = take(kCeSplitFloats * 4);
  pl->total = off;
  return LORA_OK;
}

// One-problem batch of the fused contraction with no adapter slab: out [M, N] = A [M, K] . B, B given
// as [N, K] (K-major, b_mn false) or [K, N] (MN-major, b_mn true); split when it has few tiles, with
// its partials in `part` (kCeSplitFloats elements).
// lse (fp32 output only): per-row log-sum-exp partials [M, ld_lse], written by
// the epilogue, or by the split reduce when the contraction is split.
// cand (fp32 output only): append mode instead of storing out (tau, cnt, cand,
// cap as in GemmProblem); never split.
int ce_gemm(const DeviceInfo* d, int* counter, const void* A, int64_t lda, const void* B, int64_t ldb, void* out,
            int64_t ldo, int64_t M, int64_t N, int64_t K, bool b_mn, bool f32_out, float* part, cudaStream_t st,
            float2* lse = nullptr, int ld_lse = 0, const float* tau = nullptr, int* cnt = nullptr,
            uint2* cand = nullptr, int cap = 0) {
  GemmBatch b;
  init_batch(b, d);
  b.tile_counter = counter;
  int rc;
  if ((rc = make_map(&b.tmA[0], A, K, M, lda, 64, 128)) != LORA_OK) return rc;
  b.tmA2[0] = b.tmA[0];
  if (b_mn) {
    if ((rc = make_map(&b.tmB[0], B, N, K, ldb, 64, 64)) != LORA_OK) return rc;
  } else if ((rc = make_map(&b.tmB[0], B, K, N, ldb, 64, 64)) != LORA_OK) {
    return rc;
  }
  b.tmB2[0] = b.tmB[0];
  // append mode stores nothing through the output map: a valid 32 x 32 fp32 map inside cand
  if ((rc = cand ? make_map(&b.tmOut[0], cand, 32, 32, 32, 32, 32, true)
                 : make_map(&b.tmOut[0], out, N, M, ldo, f32_out ? 32 : 64, 32, f32_out)) != LORA_OK)
    return rc;
  GemmProblem& g = b.prob[0];
  gemm_shape(g, M, N, K, 0, f32_out ? gemm_tile_n_f32() : 0);
  g.out = out;
  g.ldo = (int)ldo;
  g.out_f32 = f32_out ? 1 : 0;
  g.lse = lse;
  g.ld_lse = ld_lse;
  g.tau = tau;
  g.cnt = cnt;
  g.cand = cand;
  g.cap = cap;
  add_problem(b);
  // bf16 output with few tiles (the dh contraction of a reduced vocabulary): cut within clusters
  if (!f32_out && use_cluster_split(b, b_mn, d->num_sms / 2))
    return launch_fused_gemm_cs(b, b_mn, st) == cudaSuccess ? LORA_OK : LORA_ECUDA;
  int sp[1];
  choose_splits(b, sp);
  if (cand) sp[0] = 1;
  float* parts[1] = {part};
  if ((rc = apply_splits(b, sp, parts)) != LORA_OK) return rc;
  if (launch_fused_gemm(b, b_mn, false, d->num_sms, st, f32_out) != cudaSuccess) return LORA_ECUDA;
  return launch_split_reduce(b, st) == cudaSuccess ? LORA_OK : LORA_ECUDA;
}


// Upper triangle of the similarities of rows [r0, r0 + rows) (a whole number of
// 512-row blocks, at most 8, but for the last rows of V) in append mode: block
// I contracts against tokens from 512 I on, so its first 512-column tile is
// the diagonal block (row side only) and the others also append to the
// columns' lists.
int topk_sym_gemm(const DeviceInfo* d, int* counter, const bf* en, int64_t dd, int64_t V, int64_t r0, int64_t rows,
                  const float* tau, int* cnt, uint2* cand, int cap, cudaStream_t st) {
  GemmBatch b;
  init_batch(b, d);
  b.tile_counter = counter;
  int rc;
  for (int64_t a0 = r0; a0 < r0 + rows; a0 += kSymRows) {
    const int p = b.num_problems;
    const int64_t m = std::min<int64_t>(kSymRows, r0 + rows - a0), N = V - a0;
    if ((rc = make_map(&b.tmA[p], en + a0 * dd, dd, m, dd, 64, 128)) != LORA_OK) return rc;
    if ((rc = make_map(&b.tmB[p], en + a0 * dd, dd, N, dd, 64, 64)) != LORA_OK) return rc;
    b.tmA2[p] = b.tmA[p];
    b.tmB2[p] = b.tmB[p];
    if ((rc = make_map(&b.tmOut[p], cand, 32, 32, 32, 32, 32, true)) != LORA_OK) return rc;  // never stored through
    GemmProblem& g = b.prob[p];
    gemm_shape(g, m, N, dd, 0, gemm_tile_n_f32());
    g.out_f32 = 1;
    g.tau = tau;
    g.cnt = cnt;
    g.cand = cand;
    g.cap = cap;
    g.row_off = (int)a0;
    g.col_off = (int)a0;
    g.sym = 1;
    add_problem(b);
  }
  return launch_fused_gemm(b, false, false, d->num_sms, st, true) == cudaSuccess ? LORA_OK : LORA_ECUDA;
}

// ------------------------------------------------------------------ top-k similarity table
constexpr int kTopkChunk = 512;         // rows of materialised similarities per contraction
constexpr int kTopkSampleRows = 8192;   // rows per sample contraction
constexpr int kTopkAppendRows = 4096;   // rows per appending contraction

struct TopkPlan {
  size_t counters, status, fail_count, big_count, cnt, en, s, part, es, zs, tau, cand, fail_rows, big_rows, total;
  int chunks;                 // materialised chunks (short rows)
  int sblocks, achunks, fmax;  // sampled path: sample blocks, appending chunks, fallback batches at most
  bool sampled;
  long long lds;
};

int topk_check(const lora_bf16* E, int64_t V, int64_t d, int64_t k, TopkPlan* pl) {
  if (V < 1 || d < 8 || (d % 8) || k < 1 || k > V || k > topk_max_k() || V > (1ll << 24) || d > (1ll << 20))
    return LORA_EINVAL;
  if (E && !aligned16(E)) return LORA_EALIGN;
  pl->sampled = V >= topk_sample_min_v();
  pl->chunks = (int)cdiv(V, kTopkChunk);
  pl->sblocks = pl->sampled ? (int)cdiv(V, kTopkSampleRows) : 0;
  pl->achunks = pl->sampled ? (int)cdiv(V, kTopkAppendRows) : 0;
  pl->fmax = pl->sampled ? pl->chunks : 0;
  pl->lds = rup(V, 4);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += up256(bytes);
    return o;
  };
  // zeroed at the start of a call: tile counters, status, fallback count, candidate counts
  const int nctr = pl->sampled ? pl->sblocks + pl->achunks + pl->fmax : pl->chunks;
  pl->counters = take((size_t)nctr * 4);
  pl->status = take(4);
  pl->fail_count = take(4);
  pl->big_count = take(4);
  pl->cnt = take(pl->sampled ? (size_t)V * 4 : 0);
  pl->en = take((size_t)V * d * 2);
  pl->s = take((size_t)std::min<int64_t>(V, kTopkChunk) * pl->lds * 4);
  pl->part = take(kCeSplitFloats * 4);  // short rows: few tiles per chunk
  pl->es = pl->zs = pl->tau = pl->cand = pl->fail_rows = pl->big_rows = 0;
  if (pl->sampled) {
    pl->es = take((size_t)topk_sample() * d * 2);  // later the gathered rows of a fallback batch
    pl->zs = take((size_t)std::min<int64_t>(V, kTopkSampleRows) * topk_sample() * 4);
    pl->tau = take((size_t)V * 4);
    pl->cand = take((size_t)V * topk_cap() * 8);  // every row's list: the transposed side fills later rows
    pl->fail_rows = take((size_t)V * 4);
    pl->big_rows = take((size_t)V * 4);
  }
  pl->total = off;
  return LORA_OK;
}

}  // namespace

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// Code the calling thread's most recent entry point returned (lora_last_error).
thread_local int t_last_error = LORA_OK;
inline int rec(int rc) {
  t_last_error = rc;
  return rc;
}

bool pdl_enabled() {
  static const bool on = [] {
    const char* e = getenv("LORA_PDL");
    return !(e && e[0] == '0' && e[1] == 0);
  }();
  return on;
}

}  // namespace lora

using namespace lora;

extern "C" {

int lora_version(void) { return 300; }

int lora_last_error(void) { return t_last_error; }

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
    case LORA_ESCRATCH: return "shape needs more scratch than the fixed 4 MiB array of lora_linear_fwd_noalloc";
    default: return "unknown error";
  }
}

int lora_set_wait_limit_ns(int64_t ns) {
  std::lock_guard<std::mutex> lk(g_mu);
  g_wait_limit_ns = ns > 0 ? (long long)ns : kDefaultWaitNs;
  return rec(LORA_OK);
}

int lora_workspace_size(const lora_shape* shape, int mode, size_t* bytes) {
  if (!shape || !bytes) return rec(LORA_ENULL);
  if (mode < LORA_FWD || mode > LORA_FWD_BWD) return rec(LORA_EINVAL);
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  return rec(lora_stack_workspace_size(&p, 1, mode, bytes));
}

int lora_stack_workspace_size(const lora_proj* projs, int n_proj, int mode, size_t* bytes) {
  if (!projs || !bytes) return rec(LORA_ENULL);
  if (n_proj < 1 || n_proj > 64 || mode < LORA_FWD || mode > LORA_FWD_BWD) return rec(LORA_EINVAL);
  Plan pl;
  int rc = plan_all(projs, n_proj, mode, &pl);
  if (rc != LORA_OK) return rec(rc);
  *bytes = pl.total;
  return rec(LORA_OK);
}

namespace {
int stack_step(const lora_proj* projs, int n_proj, int mode, void* workspace, size_t workspace_bytes, void* stream,
               bool dy_cut_device);
}

int lora_stack_step(const lora_proj* projs, int n_proj, int mode, void* workspace, size_t workspace_bytes,
                    void* stream) {
  return stack_step(projs, n_proj, mode, workspace, workspace_bytes, stream, false);
}

namespace {
int stack_step(const lora_proj* projs, int n_proj, int mode, void* workspace, size_t workspace_bytes, void* stream,
               bool dy_cut_device) {
  if (!projs) return rec(LORA_ENULL);
  if (n_proj < 1 || n_proj > 64 || mode < LORA_FWD || mode > LORA_FWD_BWD) return rec(LORA_EINVAL);
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != LORA_OK) return rec(rc);
  Plan pl;
  if ((rc = plan_all(projs, n_proj, mode, &pl)) != LORA_OK) return rec(rc);
  const size_t need = pl.total;
  for (int i = 0; i < n_proj; ++i) {
    if ((mode & LORA_FWD) && (rc = check_fwd_ptrs(projs[i])) != LORA_OK) return rec(rc);
    if ((mode & LORA_BWD) && (rc = check_bwd_ptrs(projs[i])) != LORA_OK) return rec(rc);
    if (mode == LORA_FWD_BWD && projs[i].shape.rank > 0 && !projs[i].su)
      return rec(LORA_ENULL);  // the backward needs the saved su
  }
  if ((rc = check_ws(workspace, workspace_bytes, need)) != LORA_OK) return rec(rc);
  pl.dy_cut_device = dy_cut_device;
  return rec(run_step(projs, n_proj, mode, workspace, pl, d, static_cast<cudaStream_t>(stream)));
}
}  // namespace

int lora_linear_fwd(const lora_shape* shape, const lora_bf16* x, const lora_bf16* W, const lora_bf16* A,
                    const lora_bf16* B, lora_bf16* y, lora_bf16* su, void* workspace, size_t workspace_bytes,
                    void* stream) {
  if (!shape) return rec(LORA_ENULL);
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  p.x = x;
  p.W = W;
  p.A = A;
  p.B = B;
  p.y = y;
  p.su = su;
  return rec(lora_stack_step(&p, 1, LORA_FWD, workspace, workspace_bytes, stream));
}

int lora_linear_bwd(const lora_shape* shape, const lora_bf16* dy, const lora_bf16* x, const lora_bf16* W,
                    const lora_bf16* A, const lora_bf16* B, const lora_bf16* su, lora_bf16* dx, float* dA,
                    float* dB, void* workspace, size_t workspace_bytes, void* stream) {
  if (!shape) return rec(LORA_ENULL);
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
  return rec(lora_stack_step(&p, 1, LORA_BWD, workspace, workspace_bytes, stream));
}

int lora_linear_fwd_q4(const lora_shape* shape, const lora_bf16* x, const lora_q4_weight* Wq, const lora_bf16* A,
                       const lora_bf16* B, lora_bf16* y, lora_bf16* su, void* workspace, size_t workspace_bytes,
                       void* stream) {
  if (!shape || !Wq) return rec(LORA_ENULL);
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  p.x = x;
  p.Wq = *Wq;
  p.A = A;
  p.B = B;
  p.y = y;
  p.su = su;
  if (!p.Wq.codes || !p.Wq.params) return rec(LORA_ENULL);
  return rec(lora_stack_step(&p, 1, LORA_FWD, workspace, workspace_bytes, stream));
}

int lora_linear_bwd_q4(const lora_shape* shape, const lora_bf16* dy, const lora_bf16* x, const lora_q4_weight* Wq,
                       const lora_bf16* A, const lora_bf16* B, const lora_bf16* su, lora_bf16* dx, float* dA,
                       float* dB, void* workspace, size_t workspace_bytes, void* stream) {
  if (!shape || !Wq) return rec(LORA_ENULL);
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  p.dy = dy;
  p.x = x;
  p.Wq = *Wq;
  p.A = A;
  p.B = B;
  p.su = const_cast<lora_bf16*>(su);
  p.dx = dx;
  p.dA = dA;
  p.dB = dB;
  if (!p.Wq.codes || !p.Wq.params) return rec(LORA_ENULL);
  return rec(lora_stack_step(&p, 1, LORA_BWD, workspace, workspace_bytes, stream));
}

int64_t lora_launch_count(void) { return (int64_t)g_launches.load(); }

int lora_profile_begin_kinds(uint32_t kind_mask) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof.recs.clear();
  g_prof.next = 0;
  g_prof.mask = kind_mask;
  g_prof.on = true;
  return rec(LORA_OK);
}

int lora_profile_begin(void) { return lora_profile_begin_kinds((1u << LORA_KERNEL_KINDS) - 1u); }

int lora_profile_end(double* ms, int64_t* launches) {
  std::lock_guard<std::mutex> lk(g_prof_mu);
  if (!g_prof.on) return rec(LORA_EINVAL);
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
  return rec(rc);
}

int lora_stack_ckpt_workspace_size(const lora_proj* projs, int n_layers, int n_per_layer, size_t* bytes) {
  if (!bytes) return rec(LORA_ENULL);
  size_t sb = 0, wb = 0;
  const int rc = ckpt_layout(projs, n_layers, n_per_layer, &sb, &wb);
  if (rc != LORA_OK) return rec(rc);
  *bytes = sb + wb;
  return rec(LORA_OK);
}

int lora_stack_ckpt(const lora_proj* projs, int n_layers, int n_per_layer, void* workspace, size_t workspace_bytes,
                    void* stream) {
  size_t sb = 0, wb = 0;
  int rc = ckpt_layout(projs, n_layers, n_per_layer, &sb, &wb);
  if (rc != LORA_OK) return rec(rc);
  if ((rc = check_ws(workspace, workspace_bytes, sb + wb)) != LORA_OK) return rec(rc);
  DeviceInfo* d = nullptr;
  if ((rc = device_info(&d)) != LORA_OK) return rec(rc);
  uint8_t* su_scratch = static_cast<uint8_t*>(workspace);
  void* step_ws = su_scratch + sb;
  std::vector<lora_proj> layer;
  // every argument is checked before anything is enqueued
  for (int l = 0; l < n_layers; ++l) {
    layer_copy(projs + (size_t)l * n_per_layer, n_per_layer, su_scratch, &layer);
    for (const lora_proj& p : layer) {
      if ((rc = check_fwd_ptrs(p)) != LORA_OK) return rec(rc);
      if ((rc = check_bwd_ptrs(p)) != LORA_OK) return rec(rc);
    }
  }
  // Stage I: every layer's forward, saving nothing
  for (int l = 0; l < n_layers; ++l) {
    layer_copy(projs + (size_t)l * n_per_layer, n_per_layer, nullptr, &layer);
    if ((rc = lora_stack_step(layer.data(), n_per_layer, LORA_FWD, step_ws, wb, stream)) != LORA_OK) return rec(rc);
  }
  // Stage III: from the last layer back, re-run its forward saving su, then its backward
  for (int l = n_layers - 1; l >= 0; --l) {
    layer_copy(projs + (size_t)l * n_per_layer, n_per_layer, su_scratch, &layer);
    if ((rc = stack_step(layer.data(), n_per_layer, LORA_FWD_BWD, step_ws, wb, stream, true)) != LORA_OK) return rec(rc);
  }
  return rec(LORA_OK);
}

int lora_ce_workspace_size(const lora_ce_args* args, size_t* bytes) {
  if (!bytes) return rec(LORA_ENULL);
  CePlan pl;
  const int rc = ce_check(args, &pl);
  if (rc != LORA_OK) return rec(rc);
  *bytes = pl.total;
  return rec(LORA_OK);
}

int lora_ce_fwd_bwd(const lora_ce_args* a, void* workspace, size_t workspace_bytes, void* stream) {
  CePlan pl;
  int rc = ce_check(a, &pl);
  if (rc != LORA_OK) return rec(rc);
  if ((rc = check_ws(workspace, workspace_bytes, pl.total)) != LORA_OK) return rec(rc);
  DeviceInfo* d = nullptr;
  if ((rc = device_info(&d)) != LORA_OK) return rec(rc);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int T = (int)a->T, V = (int)a->V, D = (int)a->d;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  // tile counters, counts and vocabulary flags start at zero
  if (cudaMemsetAsync(ws, 0, pl.flags + (size_t)V, st) != cudaSuccess) return rec(LORA_ECUDA);
  CeIndex ix;
  ix.targets = a->targets;
  ix.mask = a->mask;
  ix.T = T;
  ix.V = V;
  ix.topk = a->topk;
  ix.ld_topk = a->ld_topk;
  ix.k = (int)a->k;
  ix.flags = ws + pl.flags;
  ix.J = at<int32_t>(ws, pl.J);
  ix.pos = at<int32_t>(ws, pl.pos);
  ix.tl = at<int32_t>(ws, pl.tl);
  ix.tpos = at<int32_t>(ws, pl.tpos);
  ix.ycol = at<int32_t>(ws, pl.ycol);
  ix.counts = at<int32_t>(ws, pl.counts);
  ix.seg_counts = at<int32_t>(ws, pl.segs);
  if (launch_ce_index(ix, st) != cudaSuccess) return rec(LORA_ECUDA);
  // |T_set| and |J| size the contractions
  int32_t counts[3] = {0, 0, 0};
  if (cudaMemcpyAsync(counts, ix.counts, sizeof(counts), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return rec(LORA_ECUDA);
  if (counts[2]) return rec(LORA_EINVAL);
  const int nT = counts[0], nJ = counts[1];
  if (a->counts) {
    a->counts[0] = nT;
    a->counts[1] = nJ;
  }
  float* rowloss = at<float>(ws, pl.rowloss);
  if (nT > 0) {
    bf* ht = at<bf>(ws, pl.ht);
    float* z = at<float>(ws, pl.z);
    bf* g = at<bf>(ws, pl.g);
    float2* lse_part = at<float2>(ws, pl.lse_part);
    const int ldz = (int)rup(nJ, 4), ldg = (int)rup(nJ, 8);
    int* tiles = at<int>(ws, pl.tiles);
    // J sorted ascending with |J| = V is every token in order: E serves as E_J
    const bf* ej = cb(a->E);
    bf* ejw = at<bf>(ws, pl.ej);
    if (launch_gather_rows2(cb(a->h), D, ix.tl, nT, ht, cb(a->E), D, ix.J, nJ < V ? nJ : 0, ejw, D, st) !=
        cudaSuccess)
      return rec(LORA_ECUDA);
    if (nJ < V) ej = ejw;
    {
      ProfScope ps(LORA_KERNEL_GEMM_FWD, st);
      if ((rc = ce_gemm(d, tiles, ht, D, ej, D, z, ldz, nT, nJ, D, false, true, at<float>(ws, pl.part), st, lse_part,
                        pl.ld_lse)) != LORA_OK)
        return rec(rc);
    }
    if (launch_ce_rows(lse_part, pl.ld_lse, z, ldz, nJ, ix.ycol, nT, at<float>(ws, pl.lse), rowloss, ix.tpos, T,
                       a->token_loss, a->loss, ix.counts + 5, g, ldg, d->num_sms, st) != cudaSuccess)
      return rec(LORA_ECUDA);
    if (a->dh) {
      bf* dht = at<bf>(ws, pl.dht);
      ProfScope ps(LORA_KERNEL_GEMM_BWD, st);
      if ((rc = ce_gemm(d, tiles + 1, g, ldg, ej, D, dht, D, nT, D, nJ, true, false, at<float>(ws, pl.part), st)) !=
          LORA_OK)
        return rec(rc);
    }
  }
  // with trainable positions the log-sum-exp launch's last block has written the losses
  if (nT == 0 && launch_ce_finish(rowloss, nT, ix.tpos, T, a->token_loss, a->loss, st) != cudaSuccess)
    return rec(LORA_ECUDA);
  if (a->dh && launch_scatter_rows(at<bf>(ws, pl.dht), ix.tpos, T, D, mb(a->dh), st) != cudaSuccess)
    return rec(LORA_ECUDA);
  if (a->vocab && nJ > 0 &&
      cudaMemcpyAsync(a->vocab, ix.J, (size_t)nJ * 4, cudaMemcpyDeviceToDevice, st) != cudaSuccess)
    return rec(LORA_ECUDA);
  return rec(LORA_OK);
}

int lora_topk_workspace_size(int64_t V, int64_t d, int64_t k, size_t* bytes) {
  if (!bytes) return rec(LORA_ENULL);
  TopkPlan pl;
  const int rc = topk_check(nullptr, V, d, k, &pl);
  if (rc != LORA_OK) return rec(rc);
  *bytes = pl.total;
  return rec(LORA_OK);
}

int lora_topk_table(const lora_bf16* E, int64_t V, int64_t d, int64_t k, int32_t* table, void* workspace,
                    size_t workspace_bytes, void* stream) {
  if (!E || !table) return rec(LORA_ENULL);
  TopkPlan pl;
  int rc = topk_check(E, V, d, k, &pl);
  if (rc != LORA_OK) return rec(rc);
  if ((rc = check_ws(workspace, workspace_bytes, pl.total)) != LORA_OK) return rec(rc);
  DeviceInfo* dv = nullptr;
  if ((rc = device_info(&dv)) != LORA_OK) return rec(rc);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  if (cudaMemsetAsync(ws, 0, pl.en, st) != cudaSuccess) return rec(LORA_ECUDA);  // counters, status, counts
  bf* en = at<bf>(ws, pl.en);
  float* S = at<float>(ws, pl.s);
  int* ctr = at<int>(ws, pl.counters);
  float* part = at<float>(ws, pl.part);
  const int D = (int)d;
  if (launch_normalize_rows(cb(E), (int)V, D, en, st) != cudaSuccess) return rec(LORA_ECUDA);
  if (!pl.sampled) {
    for (int c = 0; c < pl.chunks; ++c) {
      const int64_t r0 = (int64_t)c * kTopkChunk, rows = std::min<int64_t>(kTopkChunk, V - r0);
      {
        ProfScope ps(LORA_KERNEL_GEMM_FWD, st);
        if ((rc = ce_gemm(dv, ctr + c, en + r0 * d, d, en, d, S, pl.lds, rows, V, d, false, true, part, st)) !=
            LORA_OK)
          return rec(rc);
      }
      if (launch_topk_select(S, pl.lds, (int)V, (int)k, (int)r0, nullptr, (int)rows, table, dv->status, st) !=
          cudaSuccess)
        return rec(LORA_ECUDA);
    }
    return rec(LORA_OK);
  }
  // sampled path: thresholds from the similarities to the sample tokens
  bf* es = at<bf>(ws, pl.es);
  float* zs = at<float>(ws, pl.zs);
  float* tau = at<float>(ws, pl.tau);
  int* cnt = at<int>(ws, pl.cnt);
  uint2* cand = at<uint2>(ws, pl.cand);
  int32_t* fail_rows = at<int32_t>(ws, pl.fail_rows);
  int* fail_count = at<int>(ws, pl.fail_count);
  const int ns = topk_sample();
  int next = 0;
  if (launch_topk_gather_sample(en, (int)V, D, es, dv->num_sms, st) != cudaSuccess) return rec(LORA_ECUDA);
  for (int b = 0; b < pl.sblocks; ++b) {
    const int64_t r0 = (int64_t)b * kTopkSampleRows, rows = std::min<int64_t>(kTopkSampleRows, V - r0);
    {
      ProfScope ps(LORA_KERNEL_GEMM_FWD, st);
      if ((rc = ce_gemm(dv, ctr + next++, en + r0 * d, d, es, d, zs, ns, rows, ns, d, false, true, part, st)) !=
          LORA_OK)
        return rec(rc);
    }
    if (launch_topk_tau(zs, (int)V, (int)k, (int)rows, tau + r0, st) != cudaSuccess) return rec(LORA_ECUDA);
  }
  // the upper triangle of the similarities (C is symmetric), every value offered to both of
  // its rows' lists against their thresholds; then each row's list is sorted
  for (int c = 0; c < pl.achunks; ++c) {
    const int64_t r0 = (int64_t)c * kTopkAppendRows, rows = std::min<int64_t>(kTopkAppendRows, V - r0);
    ProfScope ps(LORA_KERNEL_GEMM_FWD, st);
    if ((rc = topk_sym_gemm(dv, ctr + next++, en, d, V, r0, rows, tau, cnt, cand, topk_cap(), st)) != LORA_OK)
      return rec(rc);
  }
  if (launch_topk_sort(cand, cnt, topk_cap(), (int)k, 0, (int)V, table, at<int32_t>(ws, pl.big_rows),
                       at<int>(ws, pl.big_count), fail_rows, fail_count, dv->num_sms, st) != cudaSuccess)
    return rec(LORA_ECUDA);
  // rows whose threshold left too few or too many candidates: the exact materialised path
  int nf = 0;
  if (cudaMemcpyAsync(&nf, fail_count, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return rec(LORA_ECUDA);
  for (int f0 = 0; f0 < nf; f0 += kTopkChunk) {
    const int n = std::min(kTopkChunk, nf - f0);
    if (launch_gather_rows(en, d, fail_rows + f0, n, D, es, st) != cudaSuccess) return rec(LORA_ECUDA);
    {
      ProfScope ps(LORA_KERNEL_GEMM_FWD, st);
      if ((rc = ce_gemm(dv, ctr + next++, es, d, en, d, S, pl.lds, n, V, d, false, true, part, st)) != LORA_OK)
        return rec(rc);
    }
    if (launch_topk_select(S, pl.lds, (int)V, (int)k, 0, fail_rows + f0, n, table, dv->status, st) != cudaSuccess)
      return rec(LORA_ECUDA);
  }
  return rec(LORA_OK);
}

int lora_wait_selftest(int64_t limit_ns, void* stream) {
  if (limit_ns < 1000 || limit_ns > 1000000000ll) return rec(LORA_EINVAL);
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != LORA_OK) return rec(rc);
  return launch_wait_probe(d->status, limit_ns, static_cast<cudaStream_t>(stream)) == cudaSuccess ? LORA_OK
                                                                                                    : LORA_ECUDA;
}

int lora_read_status(void* stream, int* status, int reset) {
  if (!status) return rec(LORA_ENULL);
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return rec(LORA_ECUDA);
  int v = 0;
  if (cudaMemcpyFromSymbol(&v, g_status, sizeof(int)) != cudaSuccess) return rec(LORA_ECUDA);
  if (reset) {
    const int z = 0;
    if (cudaMemcpyToSymbol(g_status, &z, sizeof(int)) != cudaSuccess) return rec(LORA_ECUDA);
  }
  *status = v == 0 ? LORA_OK : v == kStatusTopkTies ? LORA_EINVAL : LORA_ETIMEOUT;
  return rec(LORA_OK);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Forward for callers that cannot allocate.
//
// A caller running inside another framework's execution callback may not be
// allowed to allocate device memory, and a latency-bound caller may not
// afford the synchronisation of cudaMalloc; lora_linear_fwd_noalloc takes its
// scratch from the fixed array below instead of a caller workspace.  The
// array is a host-side stand-in in host code: its device address is looked
// up once per device with cudaGetSymbolAddress and passed to the kernels.
namespace lora {

constexpr size_t kNoAllocScratchBytes = (size_t)4 << 20;  // 4 MiB, held by every GPU that loads the library
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

namespace {
std::mutex g_noalloc_mu;
void* g_noalloc_addr[kMaxDevices] = {};
}  // namespace

}  // namespace lora

extern "C" int lora_linear_fwd_noalloc(const lora_shape* shape, const lora_bf16* x, const lora_bf16* W,
                                       const lora_bf16* A, const lora_bf16* B, lora_bf16* y, lora_bf16* su,
                                       void* stream) {
  if (!shape) return rec(LORA_ENULL);
  DeviceInfo* d = nullptr;
  int rc = device_info(&d);
  if (rc != LORA_OK) return rec(rc);
  lora_proj p;
  memset(&p, 0, sizeof(p));
  p.shape = *shape;
  p.x = x;
  p.W = W;
  p.A = A;
  p.B = B;
  p.y = y;
  p.su = su;
  Plan pl;
  if ((rc = plan_all(&p, 1, LORA_FWD, &pl, false)) != LORA_OK) return rec(rc);
  if ((rc = check_fwd_ptrs(p)) != LORA_OK) return rec(rc);  // argument errors first, as lora_stack_step
  if (pl.total > kNoAllocScratchBytes) return rec(LORA_ESCRATCH);
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return rec(LORA_ECUDA);
  void* scratch = nullptr;
  {
    // first call on this device (with it current): find the array's device address
    std::lock_guard<std::mutex> lk(g_noalloc_mu);
    if (g_noalloc_addr[dev] == nullptr) {
      void* a = nullptr;
      if (cudaGetSymbolAddress(&a, g_noalloc_scratch) != cudaSuccess || a == nullptr) return rec(LORA_ECUDA);
      g_noalloc_addr[dev] = a;
    }
    scratch = g_noalloc_addr[dev];
  }
  // run_step clears the part of the scratch that must start at zero
  return rec(run_step(&p, 1, LORA_FWD, scratch, pl, d, static_cast<cudaStream_t>(stream)));
}
