// csr_api.cpp -- host side of libcsr: the C ABI of include/csr.h.
//
// Owns the cache bookkeeping of section III-D (X_pre, the ordered X_chunks,
// the transient X_dyn suffix), the physical page pool (smallest free id
// first), two cache versions (the active one and the one a reconciliation
// rebuilds, Algorithm 1 / App. D), and the launch of the kernels:
//   foreground block:  one cooperative launch of the fused attention kernel
//                      (RoPE + paged append, attention, merge of split pieces)
//   rebuild block:     K1 rope_append -> K2 attention (short items) -> K3 merge
//   eviction:          K4 evict_compact
// The foreground runs on the caller's stream; the rebuild and its catch-up
// run on the low-priority stream registered with csr_set_reconciler, fed by
// the context's reconciliation thread (the host side of R_2).
#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <condition_variable>
#include <cstring>
#include <deque>
#include <mutex>
#include <queue>
#include <string>
#include <thread>
#include <vector>

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "../../include/csr.h"
#include "internal.h"

using namespace csr;

namespace {

// NVTX range around an entry point or a rebuild task (visible in profilers;
// no cost beyond a call when no tool is attached).
struct Range {
  explicit Range(const char *name) { nvtxRangePushA(name); }
  ~Range() { nvtxRangePop(); }
  Range(const Range &) = delete;
  Range &operator=(const Range &) = delete;
};

constexpr int kPartialItems = 4096;      // split partials a launch may write (per staging)
constexpr int kDefaultRebuildTiles = 16;
// Key tiles per CTA from which a foreground block takes the fused launch.
constexpr int kFusedMinTilesPerCta = 600;
constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
bool is_pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }

// Physical page pool: bit set = free; each request takes the smallest free id.
struct PagePool {
  int32_t n = 0;
  int32_t n_free = 0;
  std::vector<uint32_t> free_bits;
  std::vector<uint16_t> refs;

  void init(int32_t pages) {
    n = pages;
    n_free = pages;
    free_bits.assign(static_cast<size_t>(ceil_div(pages, 32)), 0u);
    for (int32_t i = 0; i < pages; ++i) free_bits[i >> 5] |= 1u << (i & 31);
    refs.assign(static_cast<size_t>(pages), 0);
  }
  int32_t take() {
    for (size_t w = 0; w < free_bits.size(); ++w) {
      if (free_bits[w]) {
        const int b = __builtin_ctz(free_bits[w]);
        free_bits[w] &= ~(1u << b);
        const int32_t id = static_cast<int32_t>(w * 32 + b);
        refs[id] = 1;
        --n_free;
        return id;
      }
    }
    return -1;
  }
  void share(int32_t id) { ++refs[id]; }
  void release(int32_t id) {
    if (--refs[id] == 0) {
      free_bits[id >> 5] |= 1u << (id & 31);
      ++n_free;
    }
  }
};

struct ChunkRec {
  int64_t id;
  int32_t len;
};

struct Version {
  std::vector<int32_t> pages;  // logical page -> physical page
  int64_t prefix_len = 0;
  std::vector<ChunkRec> chunks;
  int32_t suffix_len = 0;
  int64_t length() const {
    int64_t L = prefix_len + suffix_len;
    for (const auto &c : chunks) L += c.len;
    return L;
  }
  void clear() {
    pages.clear();
    prefix_len = 0;
    chunks.clear();
    suffix_len = 0;
  }
};

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor map: rows x d elements, boxes of 64 columns x box_rows rows,
// 128-byte swizzle (the layout the MMA descriptors describe).
bool encode_rows(CUtensorMap *m, void *base, uint64_t rows, uint64_t d, uint32_t box_rows) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[2] = {d, rows};
  cuuint64_t strides[1] = {d * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D bf16 tensor map over the block's queries q[n][hq][d]: box {64 columns,
// group heads, 128/group tokens} -- one 128-row packed query tile (rows t*G + g)
// per 64-column half, 128-byte-swizzled like the MMA operand; tokens past n
// read as zero.
bool encode_queries(CUtensorMap *m, const void *q, uint64_t n, uint64_t hq, uint64_t d, uint32_t group) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {d, hq, n};
  cuuint64_t strides[2] = {d * 2, hq * d * 2};
  cuuint32_t box[3] = {64, group, static_cast<cuuint32_t>(kBM / group)};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(q), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

struct Layout {  // workspace carve-out (byte offsets)
  size_t qpack[2], rb_out, part_o[2], part_scale[2], part_lse[2], pt[2], ids_out, err, sync, flags, total;
  int32_t rows_cap, max_pages;
};

bool valid_config(const csr_config *c, std::string *why) {
  auto bad = [&](const char *m) {
    if (why) *why = m;
    return false;
  };
  if (!c) return bad("config is NULL");
  if (c->num_q_heads <= 0 || c->num_kv_heads <= 0 || c->num_q_heads % c->num_kv_heads)
    return bad("num_q_heads must be a positive multiple of num_kv_heads");
  const int g = c->num_q_heads / c->num_kv_heads;
  if (!is_pow2(g) || g > kBM) return bad("num_q_heads/num_kv_heads must be a power of two <= 128");
  if (c->head_dim != 64 && c->head_dim != 128) return bad("head_dim must be 64 or 128");
  if (c->page_size != 16 && c->page_size != 32 && c->page_size != 64 && c->page_size != 128)
    return bad("page_size must be 16, 32, 64 or 128");
  if (!(c->rope_base > 1.0)) return bad("rope_base must be > 1");
  if (c->softmax_scale < 0.f) return bad("softmax_scale must be >= 0");
  if (c->max_new_tokens < 1) return bad("max_new_tokens must be >= 1");
  if (c->max_new_tokens / c->page_size + 2 > kMaxIdsPerCall)
    return bad("max_new_tokens / page_size too large for one launch");
  if (c->pool_pages < 1 || c->pool_pages > 32 * kMaxPoolWords)
    return bad("pool_pages must be in [1, 65536]");
  if (c->max_seq_tokens < 1 || c->max_seq_tokens > (1 << 24))
    return bad("max_seq_tokens must be in [1, 2^24] (positions are exact fp32 integers in RoPE)");
  if (static_cast<int64_t>(c->pool_pages) * c->num_kv_heads * c->page_size >= (1ll << 31))
    return bad("pool rows exceed the 32-bit TMA coordinate range");
  if (c->cap_tokens < 0 || c->evict_tokens < 0 || c->n_catchup < 0 || c->num_ctas < 0 ||
      c->rebuild_tiles_per_cta < 0 || c->fg_chunk_tiles < 0 || !(c->rebuild_duty >= 0.f))
    return bad("negative cap_tokens/evict_tokens/n_catchup/num_ctas/chunk tiles");
  if (c->cap_tokens > 0 && c->evict_tokens <= 0) return bad("cap_tokens needs evict_tokens > 0");
  return true;
}

Layout make_layout(const csr_config *c) {
  Layout L{};
  const int g = c->num_q_heads / c->num_kv_heads;
  // whole pairs of 128-row tiles, so the two-tile kernel never reads past a head's rows
  L.rows_cap = static_cast<int32_t>(align_up(static_cast<size_t>(c->max_new_tokens) * g, 2 * kBM));
  L.max_pages = static_cast<int32_t>(ceil_div(c->max_seq_tokens, c->page_size) + 1);
  const size_t d = static_cast<size_t>(c->head_dim);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes, kAlign);
    return o;
  };
  for (int i = 0; i < 2; ++i) L.qpack[i] = take(static_cast<size_t>(c->num_kv_heads) * L.rows_cap * d * 2);
  L.rb_out = take(static_cast<size_t>(c->max_new_tokens) * c->num_q_heads * d * 2);
  for (int i = 0; i < 2; ++i) {
    L.part_o[i] = take(static_cast<size_t>(kPartialItems) * kBM * d * 2);   // fp16
    L.part_scale[i] = take(static_cast<size_t>(kPartialItems) * kBM * 4);
    L.part_lse[i] = take(static_cast<size_t>(kPartialItems) * kBM * 4);
  }
  for (int i = 0; i < 2; ++i) L.pt[i] = take(static_cast<size_t>(L.max_pages) * 4);
  L.ids_out = take(static_cast<size_t>(L.max_pages) * 4);
  L.err = take(256);
  L.sync = take(256);
  L.flags = take(static_cast<size_t>(kPartialItems / 2) * 8 * 4);
  L.total = off;
  return L;
}

// One step of a rebuild, run in order on the low-priority stream by the
// reconciliation worker: the compaction kernel, or the recomputation of one
// chunk of the version being rebuilt.
struct ReconTask {
  EvictParams *compact = nullptr;  // compaction task (owned)
  ChunkRec ch{};                   // chunk task: recompute ch at positions pos..
  int64_t pos = 0;
  std::vector<int32_t> ids;        // pages of logical pages first_lp.. (empty: read the table)
  int32_t first_lp = 0;
};

// The secondary resource R_2 of Algorithm 1 on one GPU: a host thread that
// calls the provider and enqueues the rebuild on the low-priority stream, so
// the foreground caller never pays for it.
struct Reconciler {
  std::thread th;
  std::mutex mu;
  std::condition_variable cv;
  std::deque<ReconTask> q;
  bool busy = false, stop = false, started = false;
  csr_status err = CSR_OK;
  std::string err_msg;
};

}  // namespace

struct csr_ctx {
  csr_config cfg{};
  bool plan_only = false;
  int device = 0, num_sms = 0, group = 1, fg_grid = 1;
  Layout lay{};
  uint16_t *k_pool = nullptr, *v_pool = nullptr;
  uint8_t *ws = nullptr;
  CUtensorMap tm_q[2]{}, tm_k{}, tm_v{};
  double inv_turns[kMaxHalfDim]{};
  TurnSplit turns[kMaxHalfDim]{};     // inv_turns as fp32 hi + lo (rope.cuh)
  float scale_log2 = 0.f;
  // Arrivals the fused foreground launches have made on the workspace's
  // append counter (every CTA adds one per launch), so the next launch knows
  // its target; and the generation of the last fused launch (its partial
  // slots' flags hold it once written).
  uint32_t step_append = 0, step_gen = 0;
  StepParams step{};                  // parameter block of the last fused launch
  PagePool pool;
  Version ver[2];
  std::atomic<int> active{0};
  bool has_static = false;
  int64_t next_chunk_id = 0;
  // Algorithm 1 state
  bool reconciling = false;
  struct Buffered {
    ChunkRec ch;
    int64_t pos;
  };
  std::vector<Buffered> buffer;      // Delta X_buffer (N_catchup > 0): chunk and its position
  std::vector<int32_t> reserved_ids; // fresh ids the compaction kernel must produce
  bool ids_checked = false;
  bool ready = false;                 // the rebuild is complete (Algorithm 2's k_ready = k + 1)
  int64_t version = 0;                // active sequence version k (swaps so far)
  bool deferred_evict = false;        // a fused call reached tau_mem: evict at the truncation
  csr_stream_t deferred_stream = nullptr;
  csr_qkv_provider provider = nullptr;
  void *user = nullptr;
  cudaStream_t lo = nullptr;
  cudaEvent_t ev_fg = nullptr, ev_rb = nullptr;
  // recorded after every foreground launch while a reconciler is set: the
  // paced reconciliation thread starts a task only once it has completed
  cudaEvent_t ev_fg_done = nullptr;
  // Observed pace of the rebuild (App. D viability check): timing events at
  // the start of a reconciliation and after each of its tasks on the
  // low-priority stream, the query-key pairs enqueued there, and the result of
  // the last completed reconciliation.
  cudaEvent_t ev_rb_t0 = nullptr, ev_rb_t1 = nullptr;
  std::atomic<int64_t> rb_pairs{0};
  bool rb_timed = false;           // rb_pair_seconds holds an observation
  double rb_pair_seconds = 0.0;
  std::atomic<int64_t> launches{0};
  std::string err = "no error";
  Reconciler rw;
  // per-kernel event timing of foreground launches
  struct Timed {
    int kind;
    cudaEvent_t a, b;
  };
  bool timing = false;
  std::vector<Timed> timed;
  std::vector<cudaEvent_t> spare_events;

  template <class T> T *wsp(size_t off) { return reinterpret_cast<T *>(ws + off); }
  Version &act() { return ver[active.load()]; }
  Version &pend() { return ver[1 - active.load()]; }
  int32_t *d_pt(int slot) { return wsp<int32_t>(lay.pt[slot]); }
};

namespace {

// Errors raised on the reconciliation worker go to its own message, not to
// the context's (which belongs to the caller's thread).
thread_local std::string *t_err_sink = nullptr;

csr_status fail(csr_ctx *c, csr_status s, const std::string &msg) {
  if (t_err_sink)
    *t_err_sink = msg;
  else if (c)
    c->err = msg;
  return s;
}

csr_status cuda_fail(csr_ctx *c, cudaError_t e, const char *where) {
  return fail(c, CSR_ECUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

int64_t pages_for(const csr_ctx *c, int64_t len) { return ceil_div(len, c->cfg.page_size); }

// Key chunks per pair for a foreground three-launch block of `units` pairs
// whose longest key range is kv_max tiles: minimise a time estimate over the
// persistent grid -- waves x (tiles per item x t_tile + per-item cost) plus
// the split partials' write + merge read -- never more items than the
// partial buffer holds.
int32_t choose_fg_chunk_tiles(int64_t units, int64_t kv_max, int64_t grid, int head_dim) {
  // us per key tile per CTA, per item, per split partial (rough GB300 figures)
  const double t_tile = 1.5, t_item = 2.0, t_part = head_dim == 128 ? 0.04 : 0.02;
  const int64_t cap_items = kPartialItems / 2;
  int64_t best_c = kv_max;
  double best_t = 1e300;
  for (int64_t S = 1; S <= std::min<int64_t>(kv_max, 256); ++S) {
    const int64_t C = ceil_div(kv_max, S);
    const int64_t Se = ceil_div(kv_max, C);
    const int64_t items = units * Se;
    if (Se > 1 && items > cap_items) break;
    const int64_t waves = ceil_div(items, grid);
    const double t = waves * (C * t_tile + t_item) + (Se > 1 ? items * t_part : 0.0);
    if (t < best_t - 1e-9) {
      best_t = t;
      best_c = C;
    }
  }
  return static_cast<int32_t>(best_c);
}

// Key chunks per pair for a rebuild launch of `units` pairs whose longest key
// range is kv_max tiles: the fewest chunks of at most max_tiles tiles, so each
// CTA is short and a foreground launch waits at most one item for an SM;
// never more items than the partial buffer holds.
int32_t choose_chunk_tiles(int64_t units, int64_t kv_max, int max_tiles) {
  const int64_t cap_items = kPartialItems / 2;   // pair slots
  int64_t best_c = kv_max;
  for (int64_t S = 1; S <= std::min<int64_t>(kv_max, 256); ++S) {
    const int64_t C = ceil_div(kv_max, S);
    const int64_t Se = ceil_div(kv_max, C);
    if (Se > 1 && units * Se > cap_items) break;
    if (C <= max_tiles) return static_cast<int32_t>(C);
    best_c = C;  // the smallest chunk that still fits the partial buffer
  }
  return static_cast<int32_t>(best_c);
}

// Schedule of a fused foreground launch (StepSchedule) for a block of n tokens
// at L: units u = pair * hkv + head, unit u reading key tiles [0, K(u)).
//
// Balance: W = sum K(u) tiles on P CTAs takes T = ceil(W / P) tile-times.  A
// unit longer than T (cap_tiles when forced smaller) is first cut into equal
// key segments of at most that length; each segment s then runs for k_s
// tile-times and idles for T - k_s.  With V > P segments, exactly V - P of
// them idle at any time: the idle intervals are laid end to end on V - P + 1
// tracks of length T (an interval that crosses a track's end continues at the
// start of the next, so its segment idles at both ends and runs once in the
// middle).  The active intervals then never number more than P at a time, and
// dealing them to CTAs in order of start time (a CTA is free again when its
// interval ends) keeps every CTA's load within T.
//
// Locality: every segment advances one tile per tile-time while it runs, so
// at any time the keys in use lie within max(T - k_s) tiles of each other
// and the CTAs of one head read each key tile through L2 at about the same
// time: the cache is read about once.
//
// Merge: the pieces of a cut unit (one per active interval) other than the
// one that ends last write partial slots (consecutive per unit); the last one
// merges them.  A piece only ever waits for pieces that end earlier in the
// schedule (or at the same time on a lower CTA), and every CTA runs its
// pieces in schedule order, so the waits cannot form a cycle.
// One attempt with segments of at most seg_cap tiles: 1 = scheduled, 0 = more
// pieces or partial slots than one launch holds, -1 = not schedulable at all.
static int try_step_schedule(const std::vector<int64_t> &K, int64_t P, int64_t seg_cap, int64_t quantum,
                             StepSchedule &S) {
  S = StepSchedule{};
  const int32_t U = static_cast<int32_t>(K.size());
  int64_t W = 0;
  for (int64_t k : K) W += k;
  const int64_t T0 = ceil_div(W, P);
  struct Seg {
    int32_t u;
    int64_t j0, j1;
  };
  std::vector<Seg> seg;
  for (int32_t u = 0; u < U; ++u) {
    const int64_t m = ceil_div(K[u], seg_cap);
    for (int64_t s = 0; s < m; ++s) seg.push_back({u, s * K[u] / m, (s + 1) * K[u] / m});
  }
  const int64_t V = static_cast<int64_t>(seg.size());
  struct Pc {
    int32_t cta, level, u;
    int64_t b, j0, j1;
  };
  std::vector<Pc> pcs;
  std::vector<int32_t> depth(P, 0);
  int32_t used = 0;
  if (quantum > 0 && V > P) {
    // Least-advanced first: in steps of at most `quantum` tiles, the P
    // segments with the least progress run (ties: those already running,
    // which keep their CTA and extend their piece); a segment that stops
    // and later resumes on another CTA starts a new piece.
    std::vector<int64_t> prog(V, 0);
    std::vector<int32_t> on(P, -1), last_piece(P, -1);
    std::vector<int32_t> cand;
    int64_t t = 0;
    while (true) {
      cand.clear();
      for (int32_t v = 0; v < V; ++v)
        if (seg[v].j0 + prog[v] < seg[v].j1) cand.push_back(v);
      if (cand.empty()) break;
      std::vector<char> running(V, 0);
      for (int32_t c = 0; c < P; ++c)
        if (on[c] >= 0) running[on[c]] = 1;
      const size_t m = std::min<size_t>(cand.size(), static_cast<size_t>(P));
      std::partial_sort(cand.begin(), cand.begin() + m, cand.end(), [&](int32_t x, int32_t y) {
        if (prog[x] != prog[y]) return prog[x] < prog[y];
        if (running[x] != running[y]) return running[x] > running[y];
        return x < y;
      });
      std::vector<char> chosen(V, 0);
      int64_t step = quantum;
      for (size_t i = 0; i < m; ++i) {
        chosen[cand[i]] = 1;
        step = std::min(step, seg[cand[i]].j1 - seg[cand[i]].j0 - prog[cand[i]]);
      }
      std::vector<int32_t> next_on(P, -1);
      std::vector<char> placed(V, 0);
      for (int32_t c = 0; c < P; ++c)
        if (on[c] >= 0 && chosen[on[c]]) {
          next_on[c] = on[c];
          placed[on[c]] = 1;
        }
      int32_t c = 0;
      for (size_t i = 0; i < m; ++i) {
        const int32_t v = cand[i];
        if (placed[v]) continue;
        while (next_on[c] >= 0) ++c;
        next_on[c] = v;
      }
      for (int32_t cc = 0; cc < P; ++cc) {
        const int32_t v = next_on[cc];
        if (v < 0) continue;
        const int64_t j0 = seg[v].j0 + prog[v];
        const int32_t lp = last_piece[cc];
        if (lp >= 0 && on[cc] == v && pcs[lp].b == t) {
          pcs[lp].j1 += step;   // the segment keeps running on this CTA
          pcs[lp].b += step;
        } else {
          if (static_cast<int64_t>(pcs.size()) >= kMaxStepPieces) return 0;
          last_piece[cc] = static_cast<int32_t>(pcs.size());
          pcs.push_back({cc, depth[cc]++, seg[v].u, t + step, j0, j0 + step});
          used = std::max(used, cc + 1);
        }
        prog[v] += step;
      }
      on = next_on;
      t += step;
    }
  } else {
    struct Act {
      int64_t a, b;   // schedule times [a, b)
      int32_t v;
    };
    std::vector<Act> act;
    if (V <= P) {
      for (int32_t v = 0; v < V; ++v) act.push_back({0, seg[v].j1 - seg[v].j0, v});
    } else {
      // idle intervals laid end to end on tracks of length T0
      int64_t pos = 0;
      for (int32_t v = 0; v < V; ++v) {
        const int64_t k = seg[v].j1 - seg[v].j0, d = T0 - k;
        if (d == 0) {
          act.push_back({0, T0, v});
        } else if (pos + d <= T0) {
          if (pos > 0) act.push_back({0, pos, v});
          if (pos + d < T0) act.push_back({pos + d, T0, v});
          pos = pos + d == T0 ? 0 : pos + d;
        } else {
          act.push_back({pos + d - T0, pos, v});   // idle [pos, T0) and [0, pos + d - T0)
          pos = pos + d - T0;
        }
      }
    }
    std::sort(act.begin(), act.end(), [](const Act &x, const Act &y) {
      return x.a != y.a ? x.a < y.a : (x.b != y.b ? x.b < y.b : x.v < y.v);
    });
    // deal the intervals to CTAs in order of start time: the lowest free CTA
    std::priority_queue<std::pair<int64_t, int32_t>, std::vector<std::pair<int64_t, int32_t>>,
                        std::greater<std::pair<int64_t, int32_t>>> busy;   // (end, cta)
    std::priority_queue<int32_t, std::vector<int32_t>, std::greater<int32_t>> idle;
    for (int32_t c = 0; c < P; ++c) idle.push(c);
    std::vector<int64_t> done(V, 0);   // tiles of each segment dealt so far
    for (const Act &x : act) {
      while (!busy.empty() && busy.top().first <= x.a) {
        idle.push(busy.top().second);
        busy.pop();
      }
      if (idle.empty()) return -1;   // more than P intervals at once: not reachable
      const int32_t c = idle.top();
      idle.pop();
      busy.push({x.b, c});
      used = std::max(used, c + 1);
      if (static_cast<int64_t>(pcs.size()) >= kMaxStepPieces) return 0;
      const Seg &sg = seg[x.v];
      const int64_t j0 = sg.j0 + done[x.v];
      done[x.v] += x.b - x.a;
      pcs.push_back({c, depth[c]++, sg.u, x.b, j0, j0 + (x.b - x.a)});
    }
  }
  // pieces in CTA order, each CTA's in schedule order
  std::vector<int32_t> order(pcs.size());
  for (size_t i = 0; i < pcs.size(); ++i) order[i] = static_cast<int32_t>(i);
  std::sort(order.begin(), order.end(), [&](int32_t x, int32_t y) {
    return pcs[x].cta != pcs[y].cta ? pcs[x].cta < pcs[y].cta : pcs[x].level < pcs[y].level;
  });
  std::vector<int32_t> at(pcs.size());   // piece -> table index
  for (size_t i = 0; i < order.size(); ++i) {
    const Pc &pc = pcs[order[i]];
    at[order[i]] = static_cast<int32_t>(i);
    S.piece[i] = static_cast<uint64_t>(pc.u) | (static_cast<uint64_t>(pc.j0) << 16) |
                 (static_cast<uint64_t>(pc.j1) << 40);
    S.slot[i] = kSlotNone;
    S.merges[i] = 0;
    S.share[i] = 0;
  }
  for (int32_t c = 0, i = 0; c <= used; ++c) {
    while (i < static_cast<int32_t>(order.size()) && pcs[order[i]].cta < c) ++i;
    S.first[c] = static_cast<uint16_t>(i);
  }
  // per unit: the pieces that end last (its last group) merge the others.  A
  // group of one, or a unit of at most three pieces: its last member (then
  // highest CTA) combines the others' partials with its own rows.  A larger
  // group of g pieces running at the same time: all write partials and each
  // merges 256 / g of the rows over every partial, so that no single CTA
  // reads them all.
  std::vector<std::vector<int32_t>> of_unit(U);
  for (int32_t i = 0; i < static_cast<int32_t>(pcs.size()); ++i) of_unit[pcs[i].u].push_back(i);
  int32_t next = 0;
  for (int32_t u = 0; u < U; ++u) {
    auto &v = of_unit[u];
    if (v.empty()) return -1;
    if (v.size() == 1) continue;
    std::sort(v.begin(), v.end(), [&](int32_t x, int32_t y) {
      return pcs[x].b != pcs[y].b ? pcs[x].b < pcs[y].b : pcs[x].cta < pcs[y].cta;
    });
    const int32_t cnt = static_cast<int32_t>(v.size());
    int32_t g = 0;
    while (g < cnt && pcs[v[cnt - 1 - g]].b == pcs[v[cnt - 1]].b) ++g;
    if (cnt <= 3) g = 1;
    const int32_t parts = g == 1 ? cnt - 1 : cnt;
    if (next + parts > kPartialItems / 2) return 0;
    for (int32_t k = 0; k < cnt - g; ++k) S.slot[at[v[k]]] = static_cast<uint16_t>(next + k);
    if (g == 1) {
      S.slot[at[v[cnt - 1]]] = static_cast<uint16_t>(next);
      S.merges[at[v[cnt - 1]]] = static_cast<uint16_t>(parts);
      S.share[at[v[cnt - 1]]] = static_cast<uint16_t>(1 << 8);
    } else {
      for (int32_t k = 0; k < g; ++k) {
        const int32_t i = at[v[cnt - g + k]];
        S.slot[i] = static_cast<uint16_t>(next + cnt - g + k);
        S.merges[i] = static_cast<uint16_t>(parts);
        S.share[i] = static_cast<uint16_t>(k | (g << 8));
      }
    }
    next += parts;
  }
  S.grid = used;
  S.n_units = U;
  S.n_pieces = static_cast<int32_t>(pcs.size());
  S.n_slots = next;
  return 1;
}

// Key tiles per step of the least-advanced-first schedule (on request): the
// keys in use at any time stay within about this many tiles of each other
// (8 MB per head at d = 128), at the cost of a cut wherever a segment stops
// and resumes on another CTA.
constexpr int64_t kStepQuantum = 128;
int64_t step_quantum(const csr_config &cf) { return (cf.flags & CSR_FLAG_SCHEDULE_LOCAL) ? kStepQuantum : 0; }

// The schedule of a block; a forced piece length (cap_tiles > 0) grows by
// halves while the launch would hold more pieces or slots than it can.
bool build_step_schedule(int64_t L, int32_t n, int T, int hkv, int32_t n_tiles, int grid_cap,
                         int cap_tiles, int64_t quantum, StepSchedule &S) {
  const int32_t pairs = static_cast<int32_t>(ceil_div(n_tiles, 2));
  const int32_t U = pairs * hkv;
  if (U < 1 || U > 0xffff || grid_cap < 1) return false;
  std::vector<int64_t> K(U);
  int64_t W = 0;
  for (int32_t u = 0; u < U; ++u) {
    K[u] = unit_iters(L, n, T, 2 * (u / hkv) + 1);
    W += K[u];
  }
  if (K[U - 1] >= (1ll << 24)) return false;
  const int64_t P = std::min<int64_t>(grid_cap, kMaxStepGrid);
  const int64_t T0 = ceil_div(W, P);
  int64_t cap = cap_tiles > 0 ? std::min<int64_t>(T0, cap_tiles) : T0;
  while (true) {
    const int r = try_step_schedule(K, P, cap, 0, S);
    if (r == -1) return false;
    if (r == 1) break;
    if (cap >= T0) return false;
    cap = std::min(T0, cap + std::max<int64_t>(1, cap / 2));
  }
  // The least-advanced-first steps where they keep the load within 1 % of
  // the idle-interval schedule's (the optimum) and cut at most twice as often:
  // units of about equal length, a little more than one per CTA.
  if (quantum > 0) {
    static thread_local StepSchedule S2;
    if (try_step_schedule(K, P, cap, quantum, S2) == 1) {
      auto max_load = [](const StepSchedule &X) {
        int64_t m = 0;
        for (int32_t c = 0; c < X.grid; ++c) {
          int64_t l = 0;
          for (int32_t i = X.first[c]; i < X.first[c + 1]; ++i)
            l += static_cast<int64_t>((X.piece[i] >> 40) & 0xffffffu) - static_cast<int64_t>((X.piece[i] >> 16) & 0xffffffu);
          m = std::max(m, l);
        }
        return m;
      };
      const int64_t l1 = max_load(S), l2 = max_load(S2);
      if (l2 * 100 <= l1 * 101 && S2.n_slots <= 2 * S.n_slots + 8) S = S2;
    }
  }
  return true;
}

cudaEvent_t take_event(csr_ctx *c) {
  if (!c->spare_events.empty()) {
    cudaEvent_t e = c->spare_events.back();
    c->spare_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Launch through `fn` (returns cudaError_t); bracket it with timing events on
// foreground launches while timing is enabled.
template <class F>
cudaError_t timed_launch(csr_ctx *c, int kind, bool foreground, cudaStream_t s, F fn) {
  if (!(foreground && c->timing)) return fn();
  cudaEvent_t a = take_event(c), b = take_event(c);
  if (!a || !b) return cudaErrorMemoryAllocation;
  cudaError_t e = cudaEventRecord(a, s);
  if (e == cudaSuccess) e = fn();
  if (e == cudaSuccess) e = cudaEventRecord(b, s);
  if (e != cudaSuccess) return e;
  c->timed.push_back({kind, a, b});
  return cudaSuccess;
}

// Attend n new tokens at positions L.. of version `slot` (and append their
// keys/values).  ws 0 (foreground, the caller's stream): one cooperative
// launch of the fused kernel for long calls, else K1 -> K2 (persistent items)
// -> K3.  ws 1 (rebuild, the low-priority stream): K1 -> K2 (short items) ->
// K3.  ids/n_ids name the physical pages of
// logical pages first_lp.. (written into the device table by the launch);
// n_ids == 0 reads the device table instead.
csr_status run_block(csr_ctx *c, int slot, int ws, const void *q, const void *k, const void *v,
                     int32_t n, int64_t L, const int32_t *ids, int32_t n_ids, int32_t first_lp,
                     void *out, float *lse, cudaStream_t s) {
  const csr_config &cf = c->cfg;
  const bool fg = ws == 0;
  AttnParams ap{};
  ap.tm_q = c->tm_q[ws];
  ap.tm_k = c->tm_k;
  ap.tm_v = c->tm_v;
  ap.page_table = c->d_pt(slot);
  ap.out = static_cast<uint16_t *>(out);
  ap.lse = lse;
  ap.part_o = c->wsp<uint16_t>(c->lay.part_o[ws]);
  ap.part_scale = c->wsp<float>(c->lay.part_scale[ws]);
  ap.part_lse = c->wsp<float>(c->lay.part_lse[ws]);
  ap.err = c->wsp<uint32_t>(c->lay.err);
  ap.L = L;
  ap.n = n;
  ap.hq = cf.num_q_heads;
  ap.hkv = cf.num_kv_heads;
  ap.group = c->group;
  ap.page_size = cf.page_size;
  ap.rows_cap = c->lay.rows_cap;
  ap.n_tiles = static_cast<int32_t>(ceil_div(static_cast<int64_t>(n) * c->group, kBM));
  ap.n_pages_valid = static_cast<int32_t>(pages_for(c, L + n));
  ap.pool_pages = cf.pool_pages;
  ap.scale_log2 = c->scale_log2;
  const int T = kBM / c->group;

  // Foreground: one cooperative launch of the fused kernel when the call is
  // long enough for its fixed costs (query preparation and append before the
  // first tile, merges by the last pieces: tens of microseconds) to vanish
  // and has at most two units per CTA, else three chained launches (the
  // rebuild's path with a persistent grid).  Flags force either.
  bool fused = false;
  if (fg) {
    if (cf.flags & CSR_FLAG_FUSED_ALWAYS) {
      fused = true;
    } else if (!(cf.flags & CSR_FLAG_FUSED_NEVER)) {
      int64_t tiles = 0;
      const int64_t pairs = ceil_div(ap.n_tiles, 2);
      for (int64_t pr = 0; pr < pairs; ++pr) tiles += unit_iters(L, n, T, static_cast<int32_t>(2 * pr + 1));
      tiles *= cf.num_kv_heads;
      // and at most two units per CTA: with more, the fused schedule's units
      // drift apart in key position and read the cache through L2 less often
      // than the chunk-major items of the three launches
      fused = tiles >= static_cast<int64_t>(kFusedMinTilesPerCta) * c->fg_grid &&
              pairs * cf.num_kv_heads <= 2ll * c->fg_grid;
    }
    if (n_ids > kMaxStepIds) fused = false;   // more new pages than one fused launch names
  }
  StepParams &sp = c->step;
  if (fused && !build_step_schedule(L, n, T, cf.num_kv_heads, ap.n_tiles, c->fg_grid, cf.fg_chunk_tiles,
                                    step_quantum(cf), sp.s)) {
    if (cf.flags & CSR_FLAG_FUSED_ALWAYS)
      return fail(c, CSR_EINVAL, "block cannot be scheduled as one fused launch");
    fused = false;
  }
  if (fused) {
    ap.grid = sp.s.grid;
    sp.a = ap;
    sp.q = static_cast<const uint16_t *>(q);
    if (!encode_queries(&sp.tm_qraw, q, static_cast<uint64_t>(n), cf.num_q_heads, cf.head_dim, c->group))
      return fail(c, CSR_ECUDA, "encoding the queries' tensor map");
    sp.k = static_cast<const uint16_t *>(k);
    sp.v = static_cast<const uint16_t *>(v);
    sp.k_pool = c->k_pool;
    sp.v_pool = c->v_pool;
    sp.sync = c->wsp<uint32_t>(c->lay.sync);
    sp.flags = c->wsp<uint32_t>(c->lay.flags);
    sp.append_target = c->step_append + static_cast<uint32_t>(sp.s.grid);
    sp.gen = c->step_gen + 1 == 0 ? 1 : c->step_gen + 1;
    sp.first_lp = first_lp;
    sp.n_ids = n_ids;
    sp.new_lp = static_cast<int32_t>(L / cf.page_size);
    std::memcpy(sp.inv_turns, c->turns, sizeof(sp.inv_turns));
    for (int i = 0; i < n_ids; ++i) sp.ids[i] = ids[i];
    cudaError_t e =
        timed_launch(c, CSR_KERNEL_ATTENTION, true, s, [&] { return launch_step(sp, cf.head_dim, s); });
    if (e == cudaSuccess && c->rw.started) e = cudaEventRecord(c->ev_fg_done, s);
    if (e != cudaSuccess) return cuda_fail(c, e, "attention launch");
    c->step_append += static_cast<uint32_t>(sp.s.grid);
    c->step_gen = sp.gen;
    ++c->launches;
    return CSR_OK;
  }

  RopeAppendParams rp{};
  rp.q = static_cast<const uint16_t *>(q);
  rp.k = static_cast<const uint16_t *>(k);
  rp.v = static_cast<const uint16_t *>(v);
  rp.k_pool = c->k_pool;
  rp.v_pool = c->v_pool;
  rp.q_pack = c->wsp<uint16_t>(c->lay.qpack[ws]);
  rp.page_table = c->d_pt(slot);
  rp.err = ap.err;
  rp.pos0 = L;
  rp.n = n;
  rp.hq = cf.num_q_heads;
  rp.hkv = cf.num_kv_heads;
  rp.d = cf.head_dim;
  rp.page_size = cf.page_size;
  rp.group = c->group;
  rp.rows_cap = c->lay.rows_cap;
  rp.pool_pages = cf.pool_pages;
  rp.first_lp = first_lp;
  rp.n_ids = n_ids;
  std::memcpy(rp.inv_turns, c->turns, sizeof(rp.inv_turns));
  for (int i = 0; i < n_ids; ++i) rp.ids[i] = ids[i];

  const int64_t uph = ceil_div(ap.n_tiles, 2);
  const int64_t units = uph * cf.num_kv_heads;
  const int64_t kv_max = unit_iters(L, n, T, static_cast<int32_t>(uph * 2 - 1));
  if (fg) {
    // persistent CTAs over the items: a forced chunk length (never more items
    // than the partial buffer holds) or the cost model's
    if (cf.fg_chunk_tiles > 0) {
      const int64_t cap_units = std::max<int64_t>(1, kPartialItems / 2 / units);
      ap.chunk_tiles = static_cast<int32_t>(std::max<int64_t>(cf.fg_chunk_tiles, ceil_div(kv_max, cap_units)));
    } else {
      ap.chunk_tiles = choose_fg_chunk_tiles(units, kv_max, c->fg_grid, cf.head_dim);
    }
  } else {
    const int tpc = cf.rebuild_tiles_per_cta > 0 ? cf.rebuild_tiles_per_cta : kDefaultRebuildTiles;
    ap.chunk_tiles = choose_chunk_tiles(units, kv_max, tpc);
  }
  const int64_t n_chunks = ceil_div(kv_max, ap.chunk_tiles);
  ap.n_items = static_cast<int32_t>(n_chunks * units);
  // foreground: persistent CTAs over the items; rebuild: one item per CTA
  ap.grid = fg ? static_cast<int32_t>(std::min<int64_t>(c->fg_grid, ap.n_items)) : ap.n_items;
  cudaError_t e = timed_launch(c, CSR_KERNEL_ROPE_APPEND, fg, s, [&] { return launch_rope_append(rp, s); });
  if (e != cudaSuccess) return cuda_fail(c, e, "rope_append launch");
  ++c->launches;
  e = timed_launch(c, CSR_KERNEL_ATTENTION, fg, s, [&] { return launch_attention(ap, cf.head_dim, s); });
  if (e != cudaSuccess) return cuda_fail(c, e, "attention launch");
  ++c->launches;
  if (n_chunks > 1) {
    MergeParams mp{};
    mp.part_o = ap.part_o;
    mp.part_scale = ap.part_scale;
    mp.part_lse = ap.part_lse;
    mp.out = ap.out;
    mp.lse = lse;
    mp.L = L;
    mp.n = n;
    mp.hq = ap.hq;
    mp.hkv = ap.hkv;
    mp.group = ap.group;
    mp.n_tiles = ap.n_tiles;
    mp.chunk_tiles = ap.chunk_tiles;
    mp.d = cf.head_dim;
    mp.slots_per_row = merge_slots_per_row(n_chunks, mp.d);
    e = timed_launch(c, CSR_KERNEL_MERGE, fg, s, [&] { return launch_merge(mp, s); });
    if (e != cudaSuccess) return cuda_fail(c, e, "merge launch");
    ++c->launches;
  }
  if (fg && c->rw.started) {
    e = cudaEventRecord(c->ev_fg_done, s);
    if (e != cudaSuccess) return cuda_fail(c, e, "recording the foreground event");
  }
  return CSR_OK;
}

// ChunkSuffix: one block of n tokens whose first n_chunk are a chunk and the
// rest a suffix (the fused step).
enum class Kind { Prefix, Chunk, Suffix, ChunkSuffix };

void push_chunk_task(csr_ctx *c, ChunkRec ch, int64_t pos, bool write_ids);

csr_status add_block(csr_ctx *c, Kind kind, const void *q, const void *k, const void *v,
                     int32_t n, void *out, float *lse, cudaStream_t s, int64_t *chunk_id,
                     int32_t n_chunk = 0) {
  const bool is_chunk = kind == Kind::Chunk || kind == Kind::ChunkSuffix;
  const int32_t chunk_len = kind == Kind::ChunkSuffix ? n_chunk : n;
  if (n < 1 || n > c->cfg.max_new_tokens)
    return fail(c, CSR_EINVAL, "n must be in [1, max_new_tokens]");
  if (!c->plan_only && (!q || !k || !v || !out))
    return fail(c, CSR_EINVAL, "q, k, v and out must be device pointers");
  if (!c->plan_only) {
    for (const void *ptr : {q, k, v, static_cast<const void *>(out)})
      if (reinterpret_cast<uintptr_t>(ptr) % 16)
        return fail(c, CSR_EINVAL, "tensor pointers must be 16-byte aligned");
  }
  Version &A = c->act();
  const int64_t L = A.length();
  const int64_t new_len = L + n;
  if (new_len > c->cfg.max_seq_tokens) return fail(c, CSR_ENOMEM, "max_seq_tokens exceeded");
  const int64_t needA = pages_for(c, new_len) - static_cast<int64_t>(A.pages.size());
  const bool fork = is_chunk && c->reconciling;
  int64_t needB = 0;
  if (fork) {
    Version &B = c->pend();
    if (B.length() + chunk_len > c->cfg.max_seq_tokens)
      return fail(c, CSR_ENOMEM, "max_seq_tokens exceeded in the rebuilt version");
    needB = pages_for(c, B.length() + chunk_len) - static_cast<int64_t>(B.pages.size());
  }
  if (needA + needB > c->pool.n_free) return fail(c, CSR_ENOMEM, "page pool exhausted");
  // Reservation order (reading R4): the active version's pages for the chunk,
  // then the rebuilt version's for the forked chunk, then the active version's
  // for a fused suffix -- the order of csr_append_chunk + csr_attend_suffix.
  const int64_t needA_chunk =
      kind == Kind::ChunkSuffix
          ? std::max<int64_t>(0, pages_for(c, L + chunk_len) - static_cast<int64_t>(A.pages.size()))
          : needA;
  for (int64_t i = 0; i < needA_chunk; ++i) A.pages.push_back(c->pool.take());
  int64_t fork_pos = 0;
  if (fork) {
    Version &B = c->pend();
    fork_pos = B.length();
    for (int64_t i = 0; i < needB; ++i) B.pages.push_back(c->pool.take());
  }
  for (int64_t i = needA_chunk; i < needA; ++i) A.pages.push_back(c->pool.take());
  const int32_t first_lp = static_cast<int32_t>(L / c->cfg.page_size);
  const int32_t n_ids = static_cast<int32_t>(pages_for(c, new_len)) - first_lp;
  int64_t id = -1;
  if (is_chunk) id = c->next_chunk_id++;
  if (!c->plan_only) {
    const int slot = c->active.load();
    csr_status st = run_block(c, slot, 0, q, k, v, n, L, A.pages.data() + first_lp, n_ids,
                              first_lp, out, lse, s);
    if (st != CSR_OK) return st;
  }
  switch (kind) {
    case Kind::Prefix: A.prefix_len = n; break;
    case Kind::Chunk: A.chunks.push_back({id, n}); break;
    case Kind::Suffix: A.suffix_len = n; break;
    case Kind::ChunkSuffix:
      A.chunks.push_back({id, n_chunk});
      A.suffix_len = n - n_chunk;
      break;
  }
  if (chunk_id) *chunk_id = id;
  if (fork) {
    // Algorithm 1, Increment: fork the chunk into the rebuild (its pages in
    // the rebuilt version were reserved above).
    Version &B = c->pend();
    const int64_t pos = fork_pos;
    B.chunks.push_back({id, chunk_len});
    if (c->cfg.n_catchup > 0) {
      c->buffer.push_back({{id, chunk_len}, pos});
    } else if (!c->plan_only) {
      // N_catchup = 0: Algorithm 1's loop drains the whole buffer before the
      // swap, so each chunk that arrives while reconciling goes to R_2 at
      // once, in arrival order, after the foreground work that produced its
      // inputs.  (Deferring it to the next poll would never drain the buffer
      // while one chunk arrives per step.)
      cudaError_t e = cudaEventRecord(c->ev_fg, s);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(c->lo, c->ev_fg, 0);
      if (e != cudaSuccess) return cuda_fail(c, e, "ordering the catch-up after the foreground");
      push_chunk_task(c, {id, chunk_len}, pos, true);
    }
  }
  return CSR_OK;
}

// Release every page reference of a version and forget it.
void drop_version(csr_ctx *c, Version &V) {
  for (int32_t p : V.pages) c->pool.release(p);
  V.clear();
}

// Recompute one chunk of the pending version at positions pos.. on stream s
// (ws: staging buffers).  ids/first_lp name pages K1 writes into the device
// table (empty: it reads the table).
csr_status rebuild_chunk(csr_ctx *c, const ChunkRec &ch, int64_t pos,
                         const std::vector<int32_t> &ids, int32_t first_lp, int ws,
                         cudaStream_t s) {
  const void *q = nullptr, *k = nullptr, *v = nullptr;
  void *out = nullptr;
  if (c->provider(c->user, ch.id, ch.len, &q, &k, &v, &out) != 0 || !q || !k || !v)
    return fail(c, CSR_ESTATE, "qkv provider failed for chunk " + std::to_string(ch.id));
  return run_block(c, 1 - c->active.load(), ws, q, k, v, ch.len, pos, ids.data(),
                   static_cast<int32_t>(ids.size()), first_lp,
                   out ? out : c->wsp<void>(c->lay.rb_out), nullptr, s);
}

// Wait for an event by polling (the worker's own thread; yields between
// polls so that a foreground thread sharing the core is not starved).
cudaError_t wait_event(csr_ctx *c, cudaEvent_t ev) {
  (void)c;
  while (true) {
    const cudaError_t e = cudaEventQuery(ev);
    if (e != cudaErrorNotReady) return e;
    std::this_thread::yield();
  }
}

// Worker side of Reconciler: run tasks in order, record ev_rb after each.
void worker_main(csr_ctx *c) {
  cudaSetDevice(c->device);
  std::string msg;
  t_err_sink = &msg;
  std::unique_lock<std::mutex> lk(c->rw.mu);
  while (true) {
    c->rw.cv.wait(lk, [&] { return c->rw.stop || !c->rw.q.empty(); });
    if (c->rw.q.empty()) return;  // stop requested
    ReconTask t = std::move(c->rw.q.front());
    c->rw.q.pop_front();
    c->rw.busy = true;
    const bool skip = c->rw.err != CSR_OK;  // after a failure the rest is dropped
    lk.unlock();
    csr_status st = CSR_OK;
    msg.clear();
    const bool paced = !(c->cfg.flags & CSR_FLAG_UNPACED_REBUILD);
    if (!skip && paced) {
      // start only once the foreground work enqueued so far has finished
      const cudaError_t e = wait_event(c, c->ev_fg_done);
      if (e != cudaSuccess) st = cuda_fail(c, e, "waiting for the foreground work");
    }
    const auto t_task = std::chrono::steady_clock::now();
    if (!skip && st == CSR_OK) {
      Range range(t.compact ? "csr_rebuild_compact" : "csr_rebuild_chunk");
      if (t.compact) {
        const cudaError_t e = launch_evict(*t.compact, c->lo);
        if (e != cudaSuccess) st = cuda_fail(c, e, "evict_compact launch");
        else ++c->launches;
      } else {
        st = rebuild_chunk(c, t.ch, t.pos, t.ids, t.first_lp, 1, c->lo);
      }
      if (st == CSR_OK) {
        cudaError_t e = cudaEventRecord(c->ev_rb, c->lo);
        if (e == cudaSuccess) e = cudaEventRecord(c->ev_rb_t1, c->lo);
        // paced: one task in flight at a time
        if (e == cudaSuccess && paced) e = wait_event(c, c->ev_rb);
        if (e != cudaSuccess) st = cuda_fail(c, e, "recording the rebuild event");
        // and at most the configured share of wall time
        const float duty = c->cfg.rebuild_duty;
        if (st == CSR_OK && paced && duty > 0.f && duty < 1.f) {
          const double busy = std::chrono::duration<double>(std::chrono::steady_clock::now() - t_task).count();
          std::this_thread::sleep_for(std::chrono::duration<double>(busy * (1.0 / duty - 1.0)));
        }
      }
    }
    delete t.compact;
    lk.lock();
    if (st != CSR_OK && c->rw.err == CSR_OK) {
      c->rw.err = st;
      c->rw.err_msg = msg;
    }
    c->rw.busy = false;
    c->rw.cv.notify_all();
  }
}

void start_worker(csr_ctx *c) {
  if (c->rw.started || c->plan_only) return;
  c->rw.stop = false;
  c->rw.th = std::thread(worker_main, c);
  c->rw.started = true;
}

void stop_worker(csr_ctx *c) {
  if (!c->rw.started) return;
  {
    std::lock_guard<std::mutex> lk(c->rw.mu);
    for (auto &t : c->rw.q) delete t.compact;
    c->rw.q.clear();
    c->rw.stop = true;
  }
  c->rw.cv.notify_all();
  c->rw.th.join();
  c->rw.started = false;
}

void push_task(csr_ctx *c, ReconTask t) {
  {
    std::lock_guard<std::mutex> lk(c->rw.mu);
    c->rw.q.push_back(std::move(t));
  }
  c->rw.cv.notify_all();
}

// Enqueue the recomputation of chunk `ch` of the pending version at `pos`;
// write_ids: K1 writes the chunk's page ids (pages reserved after the
// compaction ran) into the device table.
void push_chunk_task(csr_ctx *c, ChunkRec ch, int64_t pos, bool write_ids) {
  // query-key pairs of the causal prefill of ch.len tokens at positions pos..
  c->rb_pairs += static_cast<int64_t>(ch.len) * pos + static_cast<int64_t>(ch.len) * (ch.len + 1) / 2;
  ReconTask t;
  t.ch = ch;
  t.pos = pos;
  if (write_ids) {
    const Version &B = c->pend();
    t.first_lp = static_cast<int32_t>(pos / c->cfg.page_size);
    const int64_t last = pages_for(c, pos + ch.len);
    t.ids.assign(B.pages.begin() + t.first_lp, B.pages.begin() + last);
  }
  push_task(c, std::move(t));
}

// Wait until the worker has nothing queued or running.
void wait_worker_idle(csr_ctx *c) {
  if (!c->rw.started) return;
  std::unique_lock<std::mutex> lk(c->rw.mu);
  c->rw.cv.wait(lk, [&] { return c->rw.q.empty() && !c->rw.busy; });
}

// Abort a reconciliation: drop queued work, wait for the device, give the
// rebuilt version's pages back.
void abort_reconcile(csr_ctx *c) {
  if (c->rw.started) {
    {
      std::lock_guard<std::mutex> lk(c->rw.mu);
      for (auto &t : c->rw.q) delete t.compact;
      c->rw.q.clear();
    }
    wait_worker_idle(c);
    std::lock_guard<std::mutex> lk(c->rw.mu);
    c->rw.err = CSR_OK;
    c->rw.err_msg.clear();
  }
  if (!c->plan_only && c->lo) cudaStreamSynchronize(c->lo);
  drop_version(c, c->pend());
  c->reconciling = false;
  c->ready = false;
  c->buffer.clear();
  c->reserved_ids.clear();
}

}  // namespace

// ============================================================== C ABI
extern "C" {

size_t csr_pool_bytes(const csr_config *cfg) {
  if (!valid_config(cfg, nullptr)) return 0;
  return static_cast<size_t>(cfg->pool_pages) * cfg->num_kv_heads * cfg->page_size *
         cfg->head_dim * 2;
}

size_t csr_workspace_bytes(const csr_config *cfg) {
  if (!valid_config(cfg, nullptr)) return 0;
  return make_layout(cfg).total;
}

csr_status csr_create(const csr_config *cfg, void *k_pool, void *v_pool, void *workspace,
                      csr_stream_t stream, csr_ctx **out) {
  static thread_local std::string create_err;
  if (!out) return CSR_EINVAL;
  *out = nullptr;
  std::string why;
  if (!valid_config(cfg, &why)) return CSR_EINVAL;
  csr_ctx *c = new csr_ctx();
  c->cfg = *cfg;
  c->plan_only = (cfg->flags & CSR_FLAG_PLAN_ONLY) != 0;
  c->group = cfg->num_q_heads / cfg->num_kv_heads;
  c->lay = make_layout(cfg);
  const double scale = cfg->softmax_scale > 0.f ? static_cast<double>(cfg->softmax_scale)
                                                : 1.0 / std::sqrt(static_cast<double>(cfg->head_dim));
  c->scale_log2 = static_cast<float>(scale * 1.4426950408889634);  // log2(e)
  const double two_pi = 6.283185307179586476925286766559;
  for (int i = 0; i < cfg->head_dim / 2; ++i) {
    c->inv_turns[i] = std::pow(cfg->rope_base, -2.0 * i / cfg->head_dim) / two_pi;
    c->turns[i].hi = static_cast<float>(c->inv_turns[i]);
    c->turns[i].lo = static_cast<float>(c->inv_turns[i] - static_cast<double>(c->turns[i].hi));
  }
  c->pool.init(cfg->pool_pages);
  if (!c->plan_only) {
    const uintptr_t a = reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
                        reinterpret_cast<uintptr_t>(workspace);
    if (!k_pool || !v_pool || !workspace || (a % kAlign)) {
      delete c;
      return CSR_EINVAL;
    }
    c->k_pool = static_cast<uint16_t *>(k_pool);
    c->v_pool = static_cast<uint16_t *>(v_pool);
    c->ws = static_cast<uint8_t *>(workspace);
    cudaError_t e = cudaGetDevice(&c->device);
    if (e == cudaSuccess)
      e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e == cudaSuccess) e = attn_configure(cfg->head_dim);
    if (e != cudaSuccess) {
      delete c;
      return CSR_ECUDA;
    }
    // the fused foreground launch is cooperative: at most one CTA per SM
    c->fg_grid = std::min(std::min(cfg->num_ctas > 0 ? cfg->num_ctas : c->num_sms, c->num_sms),
                          kMaxStepGrid);
    const uint64_t pool_rows = static_cast<uint64_t>(cfg->pool_pages) * cfg->num_kv_heads * cfg->page_size;
    const uint32_t kv_box = static_cast<uint32_t>(std::min(cfg->page_size, 64));
    bool ok = encode_rows(&c->tm_k, k_pool, pool_rows, cfg->head_dim, kv_box) &&
              encode_rows(&c->tm_v, v_pool, pool_rows, cfg->head_dim, kv_box);
    for (int i = 0; i < 2 && ok; ++i)
      ok = encode_rows(&c->tm_q[i], c->ws + c->lay.qpack[i],
                       static_cast<uint64_t>(cfg->num_kv_heads) * c->lay.rows_cap, cfg->head_dim, kBM);
    if (!ok) {
      delete c;
      return CSR_ECUDA;
    }
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const size_t pool_bytes = csr_pool_bytes(cfg);
    e = cudaMemsetAsync(k_pool, 0, pool_bytes, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(v_pool, 0, pool_bytes, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(workspace, 0, c->lay.total, s);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_fg, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_rb, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->ev_fg_done, cudaEventDisableTiming);
    if (e == cudaSuccess) e = cudaEventCreate(&c->ev_rb_t0);
    if (e == cudaSuccess) e = cudaEventCreate(&c->ev_rb_t1);
    if (e != cudaSuccess) {
      if (c->ev_fg) cudaEventDestroy(c->ev_fg);
      if (c->ev_rb) cudaEventDestroy(c->ev_rb);
      if (c->ev_fg_done) cudaEventDestroy(c->ev_fg_done);
      if (c->ev_rb_t0) cudaEventDestroy(c->ev_rb_t0);
      if (c->ev_rb_t1) cudaEventDestroy(c->ev_rb_t1);
      delete c;
      return CSR_ECUDA;
    }
  }
  *out = c;
  return CSR_OK;
}

void csr_destroy(csr_ctx *c) {
  if (!c) return;
  stop_worker(c);
  if (!c->plan_only) {
    if (c->lo) cudaStreamSynchronize(c->lo);
    cudaDeviceSynchronize();
    if (c->ev_fg) cudaEventDestroy(c->ev_fg);
    if (c->ev_rb) cudaEventDestroy(c->ev_rb);
    if (c->ev_fg_done) cudaEventDestroy(c->ev_fg_done);
    if (c->ev_rb_t0) cudaEventDestroy(c->ev_rb_t0);
    if (c->ev_rb_t1) cudaEventDestroy(c->ev_rb_t1);
    for (auto &t : c->timed) {
      cudaEventDestroy(t.a);
      cudaEventDestroy(t.b);
    }
    for (cudaEvent_t e : c->spare_events) cudaEventDestroy(e);
  }
  delete c;
}

csr_status csr_init_static(csr_ctx *c, const void *q, const void *k, const void *v, int32_t n,
                           void *out, float *lse, csr_stream_t stream) {
  Range range("csr_init_static");
  if (!c) return CSR_EINVAL;
  if (c->has_static) return fail(c, CSR_ESTATE, "static prefix already initialised");
  csr_status st = add_block(c, Kind::Prefix, q, k, v, n, out, lse,
                            reinterpret_cast<cudaStream_t>(stream), nullptr);
  if (st == CSR_OK) c->has_static = true;
  return st;
}

csr_status csr_append_chunk(csr_ctx *c, const void *q, const void *k, const void *v, int32_t n,
                            void *out, float *lse, csr_stream_t stream, int64_t *chunk_id) {
  Range range("csr_append_chunk");
  if (!c) return CSR_EINVAL;
  if (!c->has_static) return fail(c, CSR_ESTATE, "csr_init_static must come first");
  if (c->act().suffix_len > 0) return fail(c, CSR_ESTATE, "a suffix is live: truncate it first");
  csr_status st = add_block(c, Kind::Chunk, q, k, v, n, out, lse,
                            reinterpret_cast<cudaStream_t>(stream), chunk_id);
  if (st != CSR_OK) return st;
  // Algorithm 1, Increment: trigger the eviction at tau_mem.
  if (c->provider && c->cfg.cap_tokens > 0 && !c->reconciling &&
      c->act().length() >= c->cfg.cap_tokens)
    return csr_evict_and_reconcile(c, c->cfg.evict_tokens, stream);
  return CSR_OK;
}

csr_status csr_append_chunk_attend_suffix(csr_ctx *c, const void *q, const void *k, const void *v,
                                          int32_t n_chunk, int32_t n_suffix, void *out, float *lse,
                                          csr_stream_t stream, int64_t *chunk_id) {
  Range range("csr_append_chunk_attend_suffix");
  if (!c) return CSR_EINVAL;
  if (!c->has_static) return fail(c, CSR_ESTATE, "csr_init_static must come first");
  if (c->act().suffix_len > 0) return fail(c, CSR_ESTATE, "a suffix is live: truncate it first");
  if (n_chunk < 1 || n_suffix < 1) return fail(c, CSR_EINVAL, "n_chunk and n_suffix must be >= 1");
  if (static_cast<int64_t>(n_chunk) + n_suffix > c->cfg.max_new_tokens)
    return fail(c, CSR_EINVAL, "n_chunk + n_suffix must be <= max_new_tokens");
  csr_status st = add_block(c, Kind::ChunkSuffix, q, k, v, n_chunk + n_suffix, out, lse,
                            reinterpret_cast<cudaStream_t>(stream), chunk_id, n_chunk);
  if (st != CSR_OK) return st;
  // Algorithm 1, Increment: tau_mem reached; the eviction waits for the
  // truncation that ends this task (it needs no live suffix).
  if (c->provider && c->cfg.cap_tokens > 0 && !c->reconciling &&
      c->act().length() - c->act().suffix_len >= c->cfg.cap_tokens) {
    c->deferred_evict = true;
    c->deferred_stream = stream;
  }
  return CSR_OK;
}

csr_status csr_attend_suffix(csr_ctx *c, const void *q, const void *k, const void *v, int32_t n,
                             void *out, float *lse, csr_stream_t stream) {
  Range range("csr_attend_suffix");
  if (!c) return CSR_EINVAL;
  if (!c->has_static) return fail(c, CSR_ESTATE, "csr_init_static must come first");
  if (c->act().suffix_len > 0) return fail(c, CSR_ESTATE, "a suffix is already live");
  return add_block(c, Kind::Suffix, q, k, v, n, out, lse, reinterpret_cast<cudaStream_t>(stream),
                   nullptr);
}

csr_status csr_truncate_suffix(csr_ctx *c) {
  if (!c) return CSR_EINVAL;
  Version &A = c->act();
  if (A.suffix_len == 0) return fail(c, CSR_ESTATE, "no live suffix");
  A.suffix_len = 0;
  const int64_t keep = pages_for(c, A.length());
  while (static_cast<int64_t>(A.pages.size()) > keep) {
    c->pool.release(A.pages.back());
    A.pages.pop_back();
  }
  if (c->deferred_evict) {  // tau_mem was reached by a fused chunk + suffix call
    c->deferred_evict = false;
    if (c->provider && !c->reconciling)
      return csr_evict_and_reconcile(c, c->cfg.evict_tokens, c->deferred_stream);
  }
  return CSR_OK;
}

csr_status csr_rewind(csr_ctx *c, int64_t length) {
  if (!c) return CSR_EINVAL;
  Version &A = c->act();
  if (A.suffix_len > 0) return fail(c, CSR_ESTATE, "a suffix is live");
  if (c->reconciling) return fail(c, CSR_ESTATE, "a reconciliation is running");
  if (!c->has_static) return fail(c, CSR_ESTATE, "csr_init_static must come first");
  int64_t at = A.prefix_len;
  size_t keep = 0;
  while (at < length && keep < A.chunks.size()) at += A.chunks[keep++].len;
  if (at != length) return fail(c, CSR_EINVAL, "length is not the end of the prefix or of a chunk");
  A.chunks.resize(keep);
  const int64_t pages = pages_for(c, length);
  while (static_cast<int64_t>(A.pages.size()) > pages) {
    c->pool.release(A.pages.back());
    A.pages.pop_back();
  }
  return CSR_OK;
}

csr_status csr_set_reconciler(csr_ctx *c, csr_qkv_provider provider, void *user,
                              csr_stream_t lo_stream) {
  if (!c) return CSR_EINVAL;
  if (c->reconciling) return fail(c, CSR_EBUSY, "a reconciliation is running");
  wait_worker_idle(c);
  c->provider = provider;
  c->user = user;
  c->lo = reinterpret_cast<cudaStream_t>(lo_stream);
  if (provider) start_worker(c);
  return CSR_OK;
}

csr_status csr_evict_and_reconcile(csr_ctx *c, int32_t evict_tokens, csr_stream_t fg_stream) {
  Range range("csr_evict_and_reconcile");
  if (!c) return CSR_EINVAL;
  if (c->reconciling) return fail(c, CSR_EBUSY, "a reconciliation is already running");
  if (!c->provider) return fail(c, CSR_ESTATE, "no reconciler registered");
  if (evict_tokens < 1) return fail(c, CSR_EINVAL, "evict_tokens must be >= 1");
  Version &A = c->act();
  if (A.suffix_len > 0) return fail(c, CSR_ESTATE, "a suffix is live");
  if (A.chunks.empty()) return fail(c, CSR_ESTATE, "no chunk to evict");
  // Eq. eviction_operation: drop the oldest whole chunks until >= evict_tokens are gone.
  size_t k = 0;
  int64_t dropped = 0;
  while (k < A.chunks.size() && dropped < evict_tokens) dropped += A.chunks[k++].len;
  std::vector<ChunkRec> retained(A.chunks.begin() + k, A.chunks.end());
  int64_t new_len = A.prefix_len;
  for (const auto &ch : retained) new_len += ch.len;
  const int P = c->cfg.page_size;
  const int32_t full = static_cast<int32_t>(A.prefix_len / P);
  const int32_t tail = static_cast<int32_t>(A.prefix_len % P);
  const int64_t fresh = pages_for(c, new_len) - full;
  if (new_len > c->cfg.max_seq_tokens) return fail(c, CSR_ENOMEM, "max_seq_tokens exceeded");
  if (fresh > c->pool.n_free) return fail(c, CSR_ENOMEM, "page pool cannot hold the rebuilt version");
  EvictParams *ep = nullptr;
  if (!c->plan_only) {
    ep = new EvictParams();
    ep->n_words = static_cast<int32_t>(c->pool.free_bits.size());
    std::memcpy(ep->free_words, c->pool.free_bits.data(), c->pool.free_bits.size() * 4);
  }
  // Reserve the rebuilt version: shared full prefix pages, then the smallest free ids.
  const int act_slot = c->active.load();
  Version &B = c->ver[1 - act_slot];
  B.clear();
  B.prefix_len = A.prefix_len;
  for (int32_t i = 0; i < full; ++i) {
    c->pool.share(A.pages[i]);
    B.pages.push_back(A.pages[i]);
  }
  c->reserved_ids.clear();
  for (int64_t i = 0; i < fresh; ++i) {
    const int32_t id = c->pool.take();
    B.pages.push_back(id);
    c->reserved_ids.push_back(id);
  }
  B.chunks = retained;
  c->reconciling = true;
  c->buffer.clear();
  c->ids_checked = c->plan_only;
  c->rb_pairs = 0;
  if (c->plan_only) return CSR_OK;
  const cudaStream_t fg = reinterpret_cast<cudaStream_t>(fg_stream);
  cudaError_t e = cudaEventRecord(c->ev_fg, fg);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(c->lo, c->ev_fg, 0);
  if (e == cudaSuccess) e = cudaEventRecord(c->ev_rb_t0, c->lo);
  if (e != cudaSuccess) {
    delete ep;
    abort_reconcile(c);
    return cuda_fail(c, e, "ordering the rebuild after the foreground");
  }
  ep->old_pt = c->d_pt(act_slot);
  ep->new_pt = c->d_pt(1 - act_slot);
  ep->ids_out = c->wsp<int32_t>(c->lay.ids_out);
  ep->k_pool = c->k_pool;
  ep->v_pool = c->v_pool;
  ep->err = c->wsp<uint32_t>(c->lay.err);
  ep->full_prefix_pages = full;
  ep->prefix_tail = tail;
  ep->n_new = static_cast<int32_t>(fresh);
  ep->hkv = c->cfg.num_kv_heads;
  ep->page_size = P;
  ep->d = c->cfg.head_dim;
  ep->pool_pages = c->cfg.pool_pages;
  // Hand the rebuild to R_2: the compaction kernel, then the warm-up
  // (LLM(X_eps)): a fresh causal prefill of every retained chunk at its
  // renumbered position, reading the page table the compaction kernel wrote.
  ReconTask t;
  t.compact = ep;
  push_task(c, std::move(t));
  int64_t pos = A.prefix_len;
  for (const ChunkRec &ch : retained) {
    push_chunk_task(c, ch, pos, false);
    pos += ch.len;
  }
  return CSR_OK;
}

namespace {

// One step of Algorithm 1's Reconcile loop without the swap: surface a
// failure of R_2, check the compaction kernel's pages once the rebuild has
// finished, and while more than N_catchup chunks are buffered hand them to
// R_2.  *ready: the rebuilt version (k + 1) is complete up to at most
// N_catchup buffered chunks (Algorithm 2's k_ready = k + 1).
csr_status reconcile_progress(csr_ctx *c, csr_stream_t fg_stream, bool *ready) {
  *ready = false;
  if (!c->plan_only) {
    // R_2 is done when its queue is empty and its last launch has finished;
    // a task that failed there aborts the reconciliation here.
    bool idle = false;
    csr_status werr = CSR_OK;
    std::string wmsg;
    {
      std::lock_guard<std::mutex> lk(c->rw.mu);
      idle = c->rw.q.empty() && !c->rw.busy;
      werr = c->rw.err;
      wmsg = c->rw.err_msg;
    }
    if (!idle) return CSR_OK;
    if (werr != CSR_OK) {
      abort_reconcile(c);
      return fail(c, werr, wmsg);
    }
    const cudaError_t q = cudaEventQuery(c->ev_rb);
    if (q == cudaErrorNotReady) return CSR_OK;
    if (q != cudaSuccess) return cuda_fail(c, q, "rebuild event");
    if (!c->ids_checked) {
      // The compaction kernel's page choice must equal the host's reservation.
      const size_t cnt = c->reserved_ids.size();
      std::vector<int32_t> got(cnt);
      cudaError_t e = cnt ? cudaMemcpyAsync(got.data(), c->wsp<int32_t>(c->lay.ids_out), cnt * 4,
                                            cudaMemcpyDeviceToHost, c->lo)
                          : cudaSuccess;
      if (e == cudaSuccess) e = cudaStreamSynchronize(c->lo);
      if (e != cudaSuccess) return cuda_fail(c, e, "reading the compaction result");
      if (got != c->reserved_ids) {
        abort_reconcile(c);
        return fail(c, CSR_EDEVICE, "compaction kernel page ids differ from the host allocator");
      }
      c->ids_checked = true;
    }
  }
  // Algorithm 1: while |buffer| > N_catchup, catch up on the secondary resource.
  if (static_cast<int64_t>(c->buffer.size()) > c->cfg.n_catchup) {
    std::vector<csr_ctx::Buffered> batch;
    batch.swap(c->buffer);
    if (!c->plan_only) {
      const cudaStream_t fg = reinterpret_cast<cudaStream_t>(fg_stream);
      cudaError_t e = cudaEventRecord(c->ev_fg, fg);
      if (e == cudaSuccess) e = cudaStreamWaitEvent(c->lo, c->ev_fg, 0);
      if (e != cudaSuccess) return cuda_fail(c, e, "ordering the catch-up after the foreground");
      for (const auto &b : batch) push_chunk_task(c, b.ch, b.pos, true);
    }
    return CSR_OK;
  }
  if (!c->plan_only && c->rb_pairs > 0) {
    // Everything handed to R_2 so far has finished: its observed time per pair.
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, c->ev_rb_t0, c->ev_rb_t1) == cudaSuccess && ms > 0.f) {
      c->rb_pair_seconds = 1e-3 * ms / static_cast<double>(c->rb_pairs.load());
      c->rb_timed = true;
    }
  }
  *ready = true;
  return CSR_OK;
}

// App. D step 5: compute the remaining buffered chunks on the foreground and
// swap the active version atomically; the old version's own pages return to
// the pool (the shared prefix pages stay referenced).
csr_status reconcile_swap(csr_ctx *c, csr_stream_t fg_stream) {
  // The remainder (<= N_catchup chunks) is computed now, on the foreground.
  if (!c->buffer.empty()) {
    std::vector<csr_ctx::Buffered> rest;
    rest.swap(c->buffer);
    if (!c->plan_only) {
      const cudaStream_t fg = reinterpret_cast<cudaStream_t>(fg_stream);
      const Version &B = c->pend();
      for (const auto &b : rest) {
        const int32_t first_lp = static_cast<int32_t>(b.pos / c->cfg.page_size);
        const int64_t last = pages_for(c, b.pos + b.ch.len);
        std::vector<int32_t> ids(B.pages.begin() + first_lp, B.pages.begin() + last);
        csr_status st = rebuild_chunk(c, b.ch, b.pos, ids, first_lp, 0, fg);
        if (st != CSR_OK) {
          abort_reconcile(c);
          return st;
        }
      }
    }
  }
  const int old = c->active.load();
  c->active.store(1 - old);
  drop_version(c, c->ver[old]);
  c->reconciling = false;
  c->reserved_ids.clear();
  c->ready = false;
  ++c->version;
  return CSR_OK;
}

}  // namespace

csr_status csr_poll_swap(csr_ctx *c, csr_stream_t fg_stream, int *state) {
  Range range("csr_poll_swap");
  if (!c || !state) return CSR_EINVAL;
  if (!c->reconciling) {
    *state = CSR_RECON_IDLE;
    return CSR_OK;
  }
  *state = CSR_RECON_RUNNING;
  bool ready = false;
  csr_status st = reconcile_progress(c, fg_stream, &ready);
  c->ready = ready;
  if (st != CSR_OK || !ready) return st;
  if (c->act().suffix_len > 0) return CSR_OK;  // swap only between tasks
  st = reconcile_swap(c, fg_stream);
  if (st == CSR_OK) *state = CSR_RECON_SWAPPED;
  return st;
}

csr_status csr_check_viability(csr_ctx *c, int32_t evict_tokens, double append_tokens_per_s,
                               double pair_seconds, csr_viability *out) {
  if (!c || !out) return CSR_EINVAL;
  if (evict_tokens < 1 || !(append_tokens_per_s > 0.0))
    return fail(c, CSR_EINVAL, "evict_tokens must be >= 1 and the append rate > 0");
  if (c->reconciling) return fail(c, CSR_ESTATE, "a reconciliation is running");
  const Version &A = c->act();
  if (A.suffix_len > 0) return fail(c, CSR_ESTATE, "a suffix is live");
  if (A.chunks.empty()) return fail(c, CSR_ESTATE, "no chunk to evict");
  double cp = pair_seconds;
  int32_t measured = 0;
  if (!(cp > 0.0)) {
    if (!c->rb_timed) return fail(c, CSR_ESTATE, "no reconciliation has been observed yet");
    cp = c->rb_pair_seconds;
    measured = 1;
  }
  // The chunks csr_evict_and_reconcile would drop (Eq. eviction_operation).
  size_t k = 0;
  int64_t dropped = 0;
  while (k < A.chunks.size() && dropped < evict_tokens) dropped += A.chunks[k++].len;
  int64_t rebuilt = A.prefix_len;
  for (size_t i = k; i < A.chunks.size(); ++i) rebuilt += A.chunks[i].len;
  const int64_t active = A.length();
  const int P = c->cfg.page_size;
  const int64_t full = A.prefix_len / P;
  const int64_t fresh = pages_for(c, rebuilt) - full;
  const int64_t spare = static_cast<int64_t>(c->pool.n_free) - fresh;
  // N_buffer: the most tokens x for which both versions' new pages fit (Eq. oom_time).
  auto need = [&](int64_t x) {
    return (pages_for(c, active + x) - pages_for(c, active)) + (pages_for(c, rebuilt + x) - pages_for(c, rebuilt));
  };
  int64_t n_buffer = 0;
  if (spare > 0) {
    int64_t lo = 0, hi = std::max<int64_t>(0, static_cast<int64_t>(c->cfg.max_seq_tokens) - active);
    while (lo < hi) {
      const int64_t mid = lo + (hi - lo + 1) / 2;
      if (need(mid) <= spare) lo = mid;
      else hi = mid - 1;
    }
    n_buffer = lo;
  }
  const double E = static_cast<double>(rebuilt);
  const double pre = static_cast<double>(A.prefix_len);
  // Eq. warm-up_time through Eq. TTFT_derivation_2 with i* = |X_pre| + 1.
  const double t_warm = cp * (E - pre) * (E + pre + 1.0) / 2.0;
  const double dN = append_tokens_per_s * t_warm;
  const double t_recon = cp * dN * (2.0 * E + dN + 1.0) / 2.0;   // Eq. recon_time
  const double t_mem = static_cast<double>(n_buffer) / append_tokens_per_s;  // Eq. oom_time
  out->t_warm_s = t_warm;
  out->delta_n_tokens = dN;
  out->t_recon_s = t_recon;
  out->t_mem_s = t_mem;
  out->n_buffer_tokens = static_cast<double>(n_buffer);
  out->rebuilt_tokens = E;
  out->pair_seconds = cp;
  out->viable = (t_warm + t_recon <= t_mem) ? 1 : 0;   // Eq. recon_time_inequlity
  out->measured = measured;
  return CSR_OK;
}

csr_status csr_get_versions(csr_ctx *c, int64_t *k, int64_t *k_ready) {
  if (!c) return CSR_EINVAL;
  if (k) *k = c->version;
  if (k_ready) *k_ready = c->version + ((c->reconciling && c->ready) ? 1 : 0);
  return CSR_OK;
}

csr_status csr_route(csr_ctx *c, int64_t k_t, csr_stream_t fg_stream, int *route) {
  Range range("csr_route");
  if (!c || !route) return CSR_EINVAL;
  const int64_t k = c->version;
  if (k_t == k) {                       // Algorithm 2, case 1: sequence continuation
    *route = CSR_ROUTE_CONTINUE;
    return CSR_OK;
  }
  if (k_t < k) {                        // case 3: straggler
    *route = CSR_ROUTE_STRAGGLER;
    return CSR_OK;
  }
  if (k_t != k + 1 || !c->reconciling)
    return fail(c, CSR_EINVAL, "k_t names no version of this context");
  // case 2: the query is built on the evicted sequence k + 1
  bool ready = false;
  csr_status st = reconcile_progress(c, fg_stream, &ready);
  c->ready = ready;
  if (st != CSR_OK) return st;
  if (ready && c->act().suffix_len == 0) {   // k_t = k_ready: resource swap
    st = reconcile_swap(c, fg_stream);
    if (st != CSR_OK) return st;
    *route = CSR_ROUTE_SWAPPED;
    return CSR_OK;
  }
  *route = CSR_ROUTE_BRIDGE;            // k_t > k_ready: bridge on the active version
  return CSR_OK;
}

csr_status csr_cancel_reconcile(csr_ctx *c) {
  if (!c) return CSR_EINVAL;
  if (!c->reconciling) return fail(c, CSR_ESTATE, "no reconciliation running");
  abort_reconcile(c);
  return CSR_OK;
}

csr_status csr_wait_reconcile(csr_ctx *c, csr_stream_t fg_stream, int64_t timeout_us, int *state) {
  if (!c || !state) return CSR_EINVAL;
  const auto t0 = std::chrono::steady_clock::now();
  while (true) {
    csr_status st = csr_poll_swap(c, fg_stream, state);
    if (st != CSR_OK || *state != CSR_RECON_RUNNING) return st;
    if (c->act().suffix_len > 0 && c->buffer.empty())
      return fail(c, CSR_ESTATE, "swap waits for the live suffix to be truncated");
    const auto us = std::chrono::duration_cast<std::chrono::microseconds>(
                        std::chrono::steady_clock::now() - t0)
                        .count();
    if (us > timeout_us) return fail(c, CSR_ETIMEOUT, "reconciliation still running");
    std::this_thread::sleep_for(std::chrono::microseconds(50));
  }
}

csr_status csr_get_layout(csr_ctx *c, int which, int32_t *page_table, int32_t capacity,
                          int32_t *n_pages, int64_t *length) {
  if (!c) return CSR_EINVAL;
  if (which != CSR_VERSION_ACTIVE && which != CSR_VERSION_PENDING)
    return fail(c, CSR_EINVAL, "which must be ACTIVE or PENDING");
  if (which == CSR_VERSION_PENDING && !c->reconciling)
    return fail(c, CSR_ESTATE, "no reconciliation running");
  const Version &V = which == CSR_VERSION_ACTIVE ? c->act() : c->pend();
  const int32_t np = static_cast<int32_t>(V.pages.size());
  if (n_pages) *n_pages = np;
  if (length) *length = V.length();
  if (page_table) {
    if (capacity < np) return fail(c, CSR_EINVAL, "page_table capacity too small");
    std::copy(V.pages.begin(), V.pages.end(), page_table);
  }
  return CSR_OK;
}

csr_status csr_get_free_pages(csr_ctx *c, int32_t *ids, int32_t capacity, int32_t *count) {
  if (!c) return CSR_EINVAL;
  if (count) *count = c->pool.n_free;
  if (ids) {
    if (capacity < c->pool.n_free) return fail(c, CSR_EINVAL, "capacity too small");
    int32_t k = 0;
    for (int32_t i = 0; i < c->pool.n; ++i)
      if (c->pool.free_bits[i >> 5] & (1u << (i & 31))) ids[k++] = i;
  }
  return CSR_OK;
}

csr_status csr_get_chunks(csr_ctx *c, int which, int64_t *ids, int32_t *lens, int32_t capacity,
                          int32_t *count, int64_t *prefix_len) {
  if (!c) return CSR_EINVAL;
  if (which != CSR_VERSION_ACTIVE && which != CSR_VERSION_PENDING)
    return fail(c, CSR_EINVAL, "which must be ACTIVE or PENDING");
  if (which == CSR_VERSION_PENDING && !c->reconciling)
    return fail(c, CSR_ESTATE, "no reconciliation running");
  const Version &V = which == CSR_VERSION_ACTIVE ? c->act() : c->pend();
  const int32_t n = static_cast<int32_t>(V.chunks.size());
  if (count) *count = n;
  if (prefix_len) *prefix_len = V.prefix_len;
  if (ids || lens) {
    if (capacity < n) return fail(c, CSR_EINVAL, "capacity too small");
    for (int32_t i = 0; i < n; ++i) {
      if (ids) ids[i] = V.chunks[i].id;
      if (lens) lens[i] = V.chunks[i].len;
    }
  }
  return CSR_OK;
}

csr_status csr_device_page_table(csr_ctx *c, int which, const int32_t **ptr) {
  if (!c || !ptr) return CSR_EINVAL;
  if (c->plan_only) return fail(c, CSR_ESTATE, "plan-only context has no device memory");
  if (which == CSR_VERSION_PENDING && !c->reconciling)
    return fail(c, CSR_ESTATE, "no reconciliation running");
  const int slot = which == CSR_VERSION_ACTIVE ? c->active.load() : 1 - c->active.load();
  *ptr = c->d_pt(slot);
  return CSR_OK;
}

csr_status csr_gather_kv(csr_ctx *c, int which, int64_t pos0, int32_t n, void *k_out,
                         void *v_out, csr_stream_t stream) {
  if (!c) return CSR_EINVAL;
  if (c->plan_only) return fail(c, CSR_ESTATE, "plan-only context has no device memory");
  if (which != CSR_VERSION_ACTIVE && which != CSR_VERSION_PENDING)
    return fail(c, CSR_EINVAL, "which must be ACTIVE or PENDING");
  if (which == CSR_VERSION_PENDING && !c->reconciling)
    return fail(c, CSR_ESTATE, "no reconciliation running");
  const Version &V = which == CSR_VERSION_ACTIVE ? c->act() : c->pend();
  if (n < 1 || pos0 < 0 || pos0 + n > V.length() || !k_out || !v_out)
    return fail(c, CSR_EINVAL, "position range outside the version, or NULL output");
  GatherParams gp{};
  gp.k_pool = c->k_pool;
  gp.v_pool = c->v_pool;
  gp.page_table = c->d_pt(which == CSR_VERSION_ACTIVE ? c->active.load() : 1 - c->active.load());
  gp.k_out = static_cast<uint16_t *>(k_out);
  gp.v_out = static_cast<uint16_t *>(v_out);
  gp.err = c->wsp<uint32_t>(c->lay.err);
  gp.pos0 = pos0;
  gp.n = n;
  gp.hkv = c->cfg.num_kv_heads;
  gp.d = c->cfg.head_dim;
  gp.page_size = c->cfg.page_size;
  gp.pool_pages = c->cfg.pool_pages;
  const cudaError_t e = launch_gather(gp, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(c, e, "gather launch");
  ++c->launches;
  return CSR_OK;
}

csr_status csr_device_status(csr_ctx *c, uint32_t *flags) {
  if (!c) return CSR_EINVAL;
  if (flags) *flags = 0;
  if (c->plan_only) return CSR_OK;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(c, e, "device synchronise");
  uint32_t word = 0;
  e = cudaMemcpy(&word, c->wsp<uint32_t>(c->lay.err), 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemset(c->wsp<uint32_t>(c->lay.err), 0, 4);
  if (e != cudaSuccess) return cuda_fail(c, e, "reading the error word");
  if (flags) *flags = word;
  if (word) return fail(c, CSR_EDEVICE, "a kernel reported device error bits");
  return CSR_OK;
}

int64_t csr_kernel_launches(const csr_ctx *c) { return c ? c->launches.load() : 0; }

csr_status csr_set_timing(csr_ctx *c, int enable) {
  if (!c) return CSR_EINVAL;
  if (c->plan_only) return fail(c, CSR_ESTATE, "plan-only context launches no kernels");
  if (!enable) {
    for (auto &t : c->timed) {
      cudaEventSynchronize(t.b);
      c->spare_events.push_back(t.a);
      c->spare_events.push_back(t.b);
    }
    c->timed.clear();
  }
  c->timing = enable != 0;
  return CSR_OK;
}

csr_status csr_get_timing(csr_ctx *c, csr_timing *out) {
  if (!c || !out) return CSR_EINVAL;
  std::memset(out, 0, sizeof(*out));
  for (auto &t : c->timed) {
    float ms = 0.f;
    cudaError_t e = cudaEventSynchronize(t.b);
    if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, t.a, t.b);
    if (e != cudaSuccess) return cuda_fail(c, e, "reading kernel timing events");
    out->ms[t.kind] += ms;
    out->launches[t.kind] += 1;
    c->spare_events.push_back(t.a);
    c->spare_events.push_back(t.b);
  }
  c->timed.clear();
  return CSR_OK;
}

csr_status csr_foreground_schedule(const csr_config *cfg, int64_t L, int32_t n, int32_t grid,
                                   csr_piece *pieces, int32_t capacity, int32_t *count,
                                   int32_t *n_slots) {
  if (!count || !valid_config(cfg, nullptr) || L < 0 || n < 1 || n > cfg->max_new_tokens || grid < 0)
    return CSR_EINVAL;
  if (grid == 0) {
    if (cfg->flags & CSR_FLAG_PLAN_ONLY) return CSR_EINVAL;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return CSR_ECUDA;
    grid = sms;
  }
  grid = std::min(grid, kMaxStepGrid);
  const int group = cfg->num_q_heads / cfg->num_kv_heads;
  const int T = kBM / group;
  const int32_t n_tiles = static_cast<int32_t>(ceil_div(static_cast<int64_t>(n) * group, kBM));
  StepSchedule S;
  if (!build_step_schedule(L, n, T, cfg->num_kv_heads, n_tiles, grid, cfg->fg_chunk_tiles, step_quantum(*cfg), S))
    return CSR_EINVAL;
  // What each CTA's walker yields, in order.
  std::vector<csr_piece> out;
  for (int32_t c = 0; c < S.grid; ++c)
    for (int32_t i = S.first[c], order = 0; i < S.first[c + 1]; ++i, ++order) {
      const uint64_t e = S.piece[i];
      out.push_back({c, order, static_cast<int32_t>(e & 0xffffu), static_cast<int32_t>((e >> 16) & 0xffffffu),
                     static_cast<int32_t>((e >> 40) & 0xffffffu),
                     S.slot[i] == kSlotNone ? -1 : static_cast<int32_t>(S.slot[i]),
                     static_cast<int32_t>(S.merges[i]), static_cast<int32_t>(S.share[i] >> 8),
                     static_cast<int32_t>(S.share[i] & 0xffu)});
    }
  *count = static_cast<int32_t>(out.size());
  if (n_slots) *n_slots = S.n_slots;
  if (pieces) {
    if (capacity < *count) return CSR_ENOMEM;
    std::copy(out.begin(), out.end(), pieces);
  }
  return CSR_OK;
}

const char *csr_last_error(const csr_ctx *c) { return c ? c->err.c_str() : "NULL context"; }

}  // extern "C"
