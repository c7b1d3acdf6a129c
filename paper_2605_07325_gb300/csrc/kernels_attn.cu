// kernels_attn.cu -- causal attention of a block of new tokens over the paged
// cache (Eq. causal_attention_1..3: a_n = softmax(q_n K_{1:n}^T / sqrt(d_k)),
// o_n = a_n V_{1:n}), on the 5th-generation tensor cores of sm_103a.
//
// Work decomposition.  The rotated queries of one KV head are packed as rows
// t*G + g (token t, group member g), so one 128-row tile holds 128/G tokens of
// all G query heads that read the same keys.  A unit is a pair of consecutive
// query tiles (A, B) of one KV head; its key range is [0, L + last token of
// tile B].  One CTA runs one unit (or a piece of its key range) at a time, so
// every K/V tile it stages in shared memory feeds both query tiles.
//
// Roles (320 threads, one CTA per SM):
//   warp 8    TMA producer: K and V tiles page by page (page ids staged in
//             shared memory) into 128-byte-swizzled shared-memory stages; the
//             whole warp runs the loop and an elected lane issues the copies;
//   warp 9    MMA issuer: S_X = Q_X K^T (both operands in shared memory) and
//             O_X += P_X V (P from TMEM) for X = A, B, ordered PV_A(i),
//             S_A(i+1), PV_B(i), S_B(i+1), so the commit that publishes
//             S_X(i+1) also covers PV_X(i); the whole warp runs the loop and
//             elect.sync picks the issuing lane;
//   warps 0-7 softmax, one warpgroup per query tile: one thread per query row
//             (its TMEM lane); reads its scores with the row maximum reduced
//             by the TMEM load (tcgen05.ld.red, sm_103a), masks keys past the
//             row's position, keeps a running max with a lazy rescale of O
//             (only when the max grows by more than 2^8), writes P as bf16
//             over its own score columns, and finally normalises O and stores
//             it.  TMEM: S_A [0,128), S_B [128,256), O_A, O_B (d columns each).
//
// Two instantiations of attn_pair_kernel:
//   kStep = true: the foreground block in ONE cooperative launch of one CTA
//     per SM.  Every CTA appends a share of the new tokens' rotated keys and
//     values to the cache (a device counter tells the producers when key
//     tiles past position L may be read) and rotates each unit's queries
//     straight into the shared-memory Q tiles (no packed-query buffer).  The
//     CTAs walk a host-built table of pieces (unit, key tiles [j0, j1)):
//     pieces of a cut unit write normalised partial outputs and raise per-warp
//     flags; the unit's last piece waits for those flags and merges the
//     partials into its own rows (or, when several last pieces run at the
//     same time, each merges a share of the rows after its CTA's last piece).
//     No grid barrier: a piece only waits for pieces that end earlier in the
//     schedule, and every CTA is resident (cooperative launch).
//   kStep = false: one item (key chunk, head, pair) per CTA or a persistent
//     round-robin over items, queries read by TMA from the packed buffer that
//     K1 (rope_append_kernel) wrote; split items are merged by K3
//     (merge_kernel).  Used by the low-priority rebuild, whose CTAs must stay
//     short so that foreground launches get SMs quickly, and by the
//     no-allocation block path.
// Launches are chained by programmatic dependent launch: each kernel runs its
// setup while its predecessor finishes and waits (griddepcontrol) before its
// first global access.  Every wait (mbarriers, device counters) is bounded
// and reports CSR_DEVERR_WAIT_TIMEOUT.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <math_constants.h>

#include "../../include/csr.h"
#include "internal.h"
#include "ptx.cuh"
#include "rope.cuh"

namespace csr {

// One piece of work: key tiles [j0, j1) of a unit (head, pair).  A piece
// that is not the whole unit writes row r (0..255) of its partial output at
// row slot * 256 + r of the partial buffer; in the fused form the last piece
// of a cut unit instead merges the partials of slots slot .. slot + merges - 1
// (merges > 0) into its own rows and writes the output.
struct Seg {
  int32_t head, pair, slot, merges, share;
  int64_t j0, j1;
  bool complete;
};

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Bounded wait used only while unwinding after an abort.
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer_ns() - t0 > 100ull * 1000ull * 1000ull) return;
  }
}

// O row *= alpha in place (one TMEM load and store of the thread's lane).
template <int HD>
__device__ __forceinline__ void rescale_o(uint32_t taddr, float alpha) {
  uint32_t o[HD];
  if constexpr (HD == 128) tmem_ld128_wait(taddr, o);
  else tmem_ld64_wait(taddr, o);
#pragma unroll
  for (int c = 0; c < HD; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * alpha);
  if constexpr (HD == 128) tmem_st128(taddr, o);
  else tmem_st64(taddr, o);
  tmem_st_wait();
}

template <int HD>
__device__ __forceinline__ void load_o(uint32_t taddr, uint32_t (&o)[HD]) {
  if constexpr (HD == 128) tmem_ld128_wait(taddr, o);
  else tmem_ld64_wait(taddr, o);
}

// Predicated forms for a converged warp: only the lane with pred != 0 acts.
__device__ __forceinline__ uint32_t elect_lane() {
  uint32_t e;
  asm volatile("{\n\t.reg .pred p;\n\telect.sync _|p, 0xffffffff;\n\tselp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(e));
  return e;
}
__device__ __forceinline__ void mbar_arrive_expect_tx_if(uint32_t pred, uint64_t *bar, uint32_t bytes) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %2, 0;\n\t"
      "@p mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n\t}" ::"r"(smem_u32(bar)),
      "r"(bytes), "r"(pred)
      : "memory");
}
__device__ __forceinline__ void tma_load_2d_if(uint32_t pred, void *dst, const CUtensorMap *map,
                                               uint64_t *bar, int32_t x, int32_t y) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %5, 0;\n\t"
      "@p cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];\n\t}" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar)), "r"(pred)
      : "memory");
}

__device__ __forceinline__ void tma_load_3d_if(uint32_t pred, void *dst, const CUtensorMap *map,
                                               uint64_t *bar, int32_t x, int32_t y, int32_t z) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %6, 0;\n\t"
      "@p cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];\n\t}" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar)), "r"(pred)
      : "memory");
}

// Issue the TMA loads of one 128-key tile of `head` whose pages' physical ids
// are phys[0 .. 128/P): one 64-column box per page and column half (two
// 64-row boxes per page when P = 128).
template <int HD>
__device__ __forceinline__ void load_kv_tile_if(uint32_t pred, const AttnParams &p,
                                                const CUtensorMap *map, uint8_t *dst, uint64_t *bar,
                                                int head, const int32_t *phys) {
  const int P = p.page_size;
  const int ppt = kBN / P;
  const int seg = P < 64 ? P : 64;
  for (int pp = 0; pp < ppt; ++pp) {
    const int32_t row0 = (phys[pp] * p.hkv + head) * P;
    for (int r = 0; r < P; r += seg) {
#pragma unroll
      for (int b = 0; b < HD / 64; ++b)
        tma_load_2d_if(pred, dst + b * (kBN * 128) + (pp * P + r) * 128, map, bar, b * 64, row0 + r);
    }
  }
}

// ------------------------------------------------------------ device counters
__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t *ptr) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ptr) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_gpu(uint32_t *ptr, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(ptr), "r"(v) : "memory");
}
__device__ __forceinline__ void red_release_gpu_add(uint32_t *ptr, uint32_t v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(ptr), "r"(v) : "memory");
}
// Generic-proxy global writes of this thread become visible to later
// async-proxy (TMA) reads, and the reverse.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// Wait until the monotonic counter reaches target (wrap-safe).  Gives up after
// kWaitLimitNs, or when another role of the CTA aborted, returning false.
__device__ __forceinline__ bool wait_counter(const uint32_t *ctr, uint32_t target, uint32_t *err,
                                             volatile int *abort) {
  if (static_cast<int32_t>(ld_acquire_gpu(ctr) - target) >= 0) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    __nanosleep(100);
    if (static_cast<int32_t>(ld_acquire_gpu(ctr) - target) >= 0) return true;
    if (abort && *abort) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      atomicOr(err, CSR_DEVERR_WAIT_TIMEOUT);
      if (abort) *abort = 1;
      return false;
    }
  }
}
// Named barrier over `count` threads (id 0 is __syncthreads).
__device__ __forceinline__ void named_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// 16-byte load that bypasses L1 (data another SM wrote during this launch).
__device__ __forceinline__ float4 ld_cg_f4(const float *ptr) {
  float4 v;
  asm volatile("ld.global.cg.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "l"(ptr));
  return v;
}
__device__ __forceinline__ float ld_cg_f(const float *ptr) {
  float v;
  asm volatile("ld.global.cg.f32 %0, [%1];" : "=f"(v) : "l"(ptr));
  return v;
}
__device__ __forceinline__ float2 ld_cg_f2(const float *ptr) {
  float2 v;
  asm volatile("ld.global.cg.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "l"(ptr));
  return v;
}
// fp16 partial rows: 8, 4 or 2 values per load, converted in pairs
__device__ __forceinline__ uint4 ld_cg_u4(const void *ptr) {
  uint4 v;
  asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(ptr));
  return v;
}
__device__ __forceinline__ uint2 ld_cg_u2(const void *ptr) {
  uint2 v;
  asm volatile("ld.global.cg.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(ptr));
  return v;
}
__device__ __forceinline__ uint32_t ld_cg_u1(const void *ptr) {
  uint32_t v;
  asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(v) : "l"(ptr));
  return v;
}
__device__ __forceinline__ float2 half2_to_f2(uint32_t u) {
  __half2 h;
  memcpy(&h, &u, 4);
  return __half22float2(h);
}
__device__ __forceinline__ uint32_t f2_to_half2(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  uint32_t u;
  memcpy(&u, &h, 4);
  return u;
}

// ============================================================ configuration
// Shared memory: Q_A, Q_B, K and V stages, barriers, staged page ids; the
// fused form adds two RoPE angle tables (one per softmax warpgroup).
template <int HD>
struct PairCfg {
  static constexpr int kStages = (HD == 64) ? 4 : 2;
  static constexpr int kBoxes = HD / 64;
  static constexpr int kQBytes = kBM * HD * 2;                 // one query tile
  static constexpr int kTileBytes = kBN * HD * 2;
  static constexpr int kQOff = 0;                              // Q_A, then Q_B
  static constexpr int kKOff = 2 * kQBytes;
  static constexpr int kVOff = kKOff + kStages * kTileBytes;
  static constexpr int kBarOff = kVOff + kStages * kTileBytes;
  static constexpr int kPtOff = kBarOff + 1024;
  static constexpr int kPtStage = 512;
  static constexpr int kAngOff = kPtOff + kPtStage * 4;
  static constexpr int kAngEntries = 256;                      // (cos, sin) pairs per softmax warp
  static constexpr int kTurnOff = kAngOff + 8 * kAngEntries * 8;   // RoPE frequencies (TurnSplit[d/2])
  static constexpr int kIdsOff = kTurnOff + kMaxHalfDim * 8;       // the launch's first new page ids
  static constexpr int kSmemIds = 256;
  static constexpr int kSmem = kAngOff + 1024;                 // + alignment slack
  static constexpr int kSmemStep = kIdsOff + kSmemIds * 4 + 1024;
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kOCol = 2 * kBN;                   // O_A; O_B at kOCol + HD
};
static_assert(PairCfg<128>::kSmemStep <= 227 * 1024, "shared memory of the fused kernel");

struct PairBars {
  uint64_t q_full, q_empty;
  uint64_t k_full[4], k_empty[4], v_full[4], v_empty[4];
  uint64_t s_full[2], p_full[2], o_final[2], o_free[2];
  uint64_t drain, qraw_full;
  uint32_t tmem_base;
  int abort;
};

constexpr int kPairThreads = 320;

// Item form: the packed queries of an item's two tiles into the Q slots.
template <int HD>
__device__ __forceinline__ void item_q_issue(uint32_t leader, const AttnParams &A, uint8_t *smem, uint64_t *q_full,
                                             const Seg &seg) {
  using C = PairCfg<HD>;
  mbar_arrive_expect_tx_if(leader, q_full, 2 * C::kQBytes);
  const int32_t qrow = seg.head * A.rows_cap + seg.pair * 2 * kBM;
#pragma unroll
  for (int h = 0; h < 2; ++h)
#pragma unroll
    for (int b = 0; b < C::kBoxes; ++b)
      tma_load_2d_if(leader, smem + C::kQOff + h * C::kQBytes + b * (kBM * 128), &A.tm_q, q_full, b * 64,
                     qrow + h * kBM);
}

// ============================================================ work walkers
// Items of the non-fused form: (chunk, head, pair); the pair's key range is
// that of its second tile.
struct PairWalker {
  int32_t item;
  __device__ bool next(const AttnParams &p, int T, Seg &s) {
    const int32_t n_pairs = (p.n_tiles + 1) / 2;
    const int32_t units = p.hkv * n_pairs;
    while (item < p.n_items) {
      const int32_t it = item;
      item += p.grid;
      const int32_t k = it / units;
      const int32_t rem = it - k * units;
      const int32_t head = rem / n_pairs;
      const int32_t pair = rem - head * n_pairs;
      const int64_t kv = unit_iters(p.L, p.n, T, 2 * pair + 1);
      const int64_t j0 = static_cast<int64_t>(k) * p.chunk_tiles;
      if (j0 >= kv) continue;
      s.head = head;
      s.pair = pair;
      s.slot = it;
      s.merges = 0;
      s.share = 0;
      s.j0 = j0;
      s.j1 = min(j0 + p.chunk_tiles, kv);
      s.complete = kv <= p.chunk_tiles;
      return true;
    }
    return false;
  }
};

// Pieces of the fused form (StepSchedule); units u = pair * hkv + head.
struct StepWalker {
  int32_t i, end;
  __device__ bool next(const StepParams &p, int T, Seg &s) {
    const StepSchedule &S = p.s;
    (void)T;
    if (i >= end) return false;
    const uint64_t e = S.piece[i];
    const int32_t u = static_cast<int32_t>(e & 0xffffu);
    const int32_t pair = u / p.a.hkv;
    s.head = u - pair * p.a.hkv;
    s.pair = pair;
    s.j0 = static_cast<int64_t>((e >> 16) & 0xffffffu);
    s.j1 = static_cast<int64_t>((e >> 40) & 0xffffffu);
    s.slot = S.slot[i];
    s.merges = S.merges[i];
    s.share = S.share[i];
    s.complete = s.slot == kSlotNone;
    ++i;
    return true;
  }
};

template <bool kStep> struct PairTraits;
template <> struct PairTraits<false> {
  using Params = AttnParams;
  using Walker = PairWalker;
};
template <> struct PairTraits<true> {
  using Params = StepParams;
  using Walker = StepWalker;
};
__device__ __forceinline__ const AttnParams &attn_of(const AttnParams &p) { return p; }
__device__ __forceinline__ const AttnParams &attn_of(const StepParams &p) { return p.a; }
__device__ __forceinline__ PairWalker make_walker(const AttnParams &) {
  return PairWalker{static_cast<int32_t>(blockIdx.x)};
}
__device__ __forceinline__ StepWalker make_walker(const StepParams &p) {
  return StepWalker{p.s.first[blockIdx.x], p.s.first[blockIdx.x + 1]};
}

// ============================================================ fused-form steps
// Physical page of logical page lp of the block's version: the launch's new
// pages come from its id list (the first kSmemIds copied to shared memory at
// entry, `ids_s`), the older ones from the table.  -1 when out of range.
__device__ __forceinline__ int32_t step_page(const StepParams &p, const int32_t *ids_s, int64_t lp) {
  const AttnParams &A = p.a;
  int32_t phys;
  if (lp >= p.first_lp && lp < p.first_lp + p.n_ids) {
    phys = ids_s[lp - p.first_lp];   // n_ids <= kSmemIds
  } else {
    phys = A.page_table[lp];
  }
  return (phys < 0 || phys >= A.pool_pages) ? -1 : phys;
}

// This CTA's share of the append (nthreads threads, tid 0..nthreads-1):
// rotated keys and values of the new tokens into their cache slots, and
// (CTA 0) the new pages' ids into the device table.  Work items of 16 bytes
// out: 8 key pairs (two stores) or 8 values.
template <int HD>
__device__ __noinline__ void step_append(const StepParams &p, const TurnSplit *turns, const int32_t *ids_s, int tid,
                                         int nthreads) {
  const AttnParams &A = p.a;
  constexpr int half = HD / 2, c16 = HD / 16, c8 = HD / 8;
  constexpr int kBatch = 4;   // items whose input loads are in flight together
  if (blockIdx.x == 0) {
    int32_t *table = const_cast<int32_t *>(A.page_table);
    for (int i = tid; i < p.n_ids; i += nthreads) table[p.first_lp + i] = p.ids[i];
  }
  const int64_t nk = static_cast<int64_t>(A.n) * A.hkv * c16;
  const int64_t nv = static_cast<int64_t>(A.n) * A.hkv * c8;
  // items interleaved over the CTAs (item g = tid * grid + CTA), so a small
  // block spreads over every CTA instead of filling the first ones
  const int64_t stride = static_cast<int64_t>(gridDim.x) * nthreads;
  for (int64_t w0 = static_cast<int64_t>(tid) * gridDim.x + blockIdx.x; w0 < nk + nv; w0 += kBatch * stride) {
    uint4 a[kBatch], b[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {   // the inputs of up to four items
      const int64_t w = w0 + u * stride;
      if (w >= nk + nv) break;
      const bool is_k = w < nk;
      const int64_t ww = is_k ? w : w - nk;
      const int per_tok = A.hkv * (is_k ? c16 : c8);
      const int64_t t = ww / per_tok;
      const int rem = static_cast<int>(ww - t * per_tok);
      const int h = rem / (is_k ? c16 : c8);
      const int i0 = (rem % (is_k ? c16 : c8)) * 8;
      if (is_k) {
        const uint16_t *src = p.k + (t * A.hkv + h) * HD;
        a[u] = *reinterpret_cast<const uint4 *>(src + i0);
        b[u] = *reinterpret_cast<const uint4 *>(src + i0 + half);
      } else {
        a[u] = *reinterpret_cast<const uint4 *>(p.v + (t * A.hkv + h) * HD + i0);
      }
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const int64_t w = w0 + u * stride;
      if (w >= nk + nv) break;
      const bool is_k = w < nk;
      const int64_t ww = is_k ? w : w - nk;
      const int per_tok = A.hkv * (is_k ? c16 : c8);
      const int64_t t = ww / per_tok;
      const int rem = static_cast<int>(ww - t * per_tok);
      const int h = rem / (is_k ? c16 : c8);
      const int i0 = (rem % (is_k ? c16 : c8)) * 8;
      const int64_t pos = A.L + t;
      const int64_t lp = pos / A.page_size;
      const int32_t phys = step_page(p, ids_s, lp);
      if (phys < 0) {
        atomicOr(A.err, CSR_DEVERR_BAD_PAGE);
        continue;
      }
      const int64_t slot_row = (static_cast<int64_t>(phys) * A.hkv + h) * A.page_size + (pos - lp * A.page_size);
      if (is_k) {
        float cs[8], sn[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) rope_cos_sin(pos, turns[i0 + e], cs[e], sn[e]);
        uint4 ya, yb;
        rope_rotate8(a[u], b[u], cs, sn, ya, yb);
        uint16_t *dst = p.k_pool + slot_row * HD;
        *reinterpret_cast<uint4 *>(dst + i0) = ya;
        *reinterpret_cast<uint4 *>(dst + i0 + half) = yb;
      } else {
        *reinterpret_cast<uint4 *>(p.v_pool + slot_row * HD + i0) = a[u];
      }
    }
  }
  fence_proxy_async_global();   // the other CTAs read these slots by TMA
}

// The raw queries of a unit's two query tiles, brought by the producer: one
// 3-D TMA box {64 columns, G heads, 128/G tokens} per tile and column half,
// landing in the 128-byte-swizzled K-major layout the MMA descriptors describe
// (tile row r = token r / G, head head * G + r % G; tokens past the block read
// as zero).
template <int HD>
__device__ __forceinline__ void step_qraw_issue(uint32_t pred, const StepParams &p, uint8_t *smem,
                                                uint64_t *bar, int head, int pair, int T) {
  using C = PairCfg<HD>;
  const int G = p.a.group;
  mbar_arrive_expect_tx_if(pred, bar, 2 * C::kQBytes);
#pragma unroll
  for (int x = 0; x < 2; ++x)
#pragma unroll
    for (int b = 0; b < C::kBoxes; ++b)
      tma_load_3d_if(pred, smem + C::kQOff + x * C::kQBytes + b * (kBM * 128), &p.tm_qraw, bar, b * 64,
                     head * G, (pair * 2 + x) * T);
}

// The (cos, sin) of the tokens of this softmax warp's 32 rows (token r / G of
// tile `wg` of the pair) into the warp's table `ang`: entry (token - w0) *
// d/2 + i, tokens w0 .. w1 - 1.  Shared by the G heads of a token; only
// __syncwarp orders it.  Returns the number of tokens held (at most
// kAngEntries / (d/2)); rows of later tokens are rotated in a second batch.
template <int HD>
__device__ __forceinline__ int step_angles(const StepParams &p, float2 *ang, const TurnSplit *turns,
                                           int pair, int wg, int row, int lane, int T, int b0, int w1) {
  constexpr int half = HD / 2;
  constexpr int per_batch = PairCfg<HD>::kAngEntries / half;
  const int64_t tok0 = static_cast<int64_t>(pair * 2 + wg) * T;
  const int bt = min(per_batch, w1 - b0);
  __syncwarp();   // the previous batch's table is no longer read
  for (int e = lane; e < bt * half; e += 32) {
    const int tt = e / half;
    const int i = e - tt * half;
    float c, s;
    rope_cos_sin(p.a.L + tok0 + b0 + tt, turns[i], c, s);
    ang[e] = make_float2(c, s);
  }
  __syncwarp();
  return bt;
}

// Rotate this thread's query row in place (its own 128-byte lines of the two
// column boxes: 16-byte chunk c at position c ^ (r % 8)), with the angles of
// its token (row `ang_row` of the table); ends with the proxy fence that lets
// the tensor core read the rotated tile.
template <int HD>
__device__ __forceinline__ void step_rotate_row(uint8_t *qtile, const float2 *a, int row) {
  constexpr int c16 = HD / 16;
  uint8_t *line = qtile + row * 128;
  const uint32_t sw = static_cast<uint32_t>(row & 7);
  auto at = [&](int c) {
    return reinterpret_cast<uint4 *>(line + (c >> 3) * (kBM * 128) + ((static_cast<uint32_t>(c & 7) ^ sw) * 16));
  };
  // a rolled loop: this runs once per piece, and a short body is fetched once
#pragma unroll 1
  for (int c = 0; c < c16; ++c) {
    const uint4 xa = *at(c), xb = *at(c + c16);
    float cs[8], sn[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float2 v = a[c * 8 + e];
      cs[e] = v.x;
      sn[e] = v.y;
    }
    uint4 ya, yb;
    rope_rotate8(xa, xb, cs, sn, ya, yb);
    *at(c) = ya;
    *at(c + c16) = yb;
  }
}

// A softmax warp's share of a piece's query preparation: the angle tables of
// its tokens, then (once the raw queries are in, `qraw_parity` of the
// producer's barrier) the in-place rotation of its 32 rows, the proxy fence
// and one arrival on q_full.  Returns false if the wait gave up.
template <int HD>
__device__ __noinline__ bool step_q_prep(const StepParams &p, uint8_t *qtile, float2 *ang, const TurnSplit *turns,
                                         uint64_t *qraw_full, uint32_t qraw_parity, uint64_t *q_full,
                                         volatile int *abort, int pair, int wg, int row, int lane, int T) {
  constexpr int half = HD / 2;
  const int G = p.a.group;
  const int tr = row / G;
  const int w0 = (row - lane) / G, w1 = (row - lane + 31) / G + 1;   // the warp's tokens
  int b0 = w0;
  int bt = step_angles<HD>(p, ang, turns, pair, wg, row, lane, T, b0, w1);
  const bool got = mbar_wait(qraw_full, qraw_parity, abort, p.a.err, CSR_DEVERR_WAIT_TIMEOUT);
  if (!__all_sync(0xffffffffu, got)) return false;
  while (true) {
    if (tr >= b0 && tr < b0 + bt) step_rotate_row<HD>(qtile, ang + (tr - b0) * half, row);
    b0 += bt;
    if (b0 >= w1) break;
    bt = step_angles<HD>(p, ang, turns, pair, wg, row, lane, T, b0, w1);
  }
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) mbar_arrive(q_full);
  return true;
}

// Merge share of a member of a unit's last group (fused form, group of g > 1
// pieces that run at the same time): rows [k * 256 / g, (k + 1) * 256 / g) of
// the unit's 256, spread over the CTA's eight softmax warps, over the unit's
// cnt partial slots (every piece's normalised rows and log2-sum-exps, the group's own
// included): lse = log2 sum_k 2^lse_k, out = sum_k 2^(lse_k - lse) O_k.  One
// row per warp at a time, HD / 32 columns per lane; the flags of the warp
// that wrote the row in every piece are awaited first.  False after a failed
// wait.
template <int HD>
__device__ __noinline__ bool step_merge_share(const StepParams &p, const Seg &seg, int T, int w8, int lane,
                                              volatile int *abort) {
  const AttnParams &A = p.a;
  constexpr int kPer = HD / 32;
  const int32_t g = seg.share >> 8, k = seg.share & 0xff, cnt = seg.merges;
  const int64_t s0 = static_cast<int64_t>(seg.slot) - (cnt - g) - k;
  const int r_a = k * kPairRows / g, r_b = (k + 1) * kPairRows / g;
  int last_fw = -1;
  for (int r = r_a + w8; r < r_b; r += 8) {   // rows over all eight softmax warps
    const int tile = seg.pair * 2 + r / kBM;
    const int rr = r % kBM;
    const int64_t t = static_cast<int64_t>(tile) * T + rr / A.group;
    if (tile >= A.n_tiles || t >= A.n) continue;
    const int fw = r / 32;   // the softmax warp that wrote row r in every piece
    if (fw != last_fw) {
      bool got = true;
      for (int kk = lane; kk < cnt && got; kk += 32)
        got = wait_counter(p.flags + (s0 + kk) * 8 + fw, p.gen, A.err, abort);
      if (!__all_sync(0xffffffffu, got)) return false;
      last_fw = fw;
    }
    const float *lse_r = A.part_lse + s0 * kPairRows + r;
    // lse = log2 sum_k 2^lse_k in one pass: a running (max, sum) per lane,
    // then combined over the warp
    float mx = -CUDART_INF_F, sum = 0.f;
    for (int kk = lane; kk < cnt; kk += 32) {
      const float x = ld_cg_f(lse_r + static_cast<int64_t>(kk) * kPairRows);
      if (x > mx) {
        sum = (mx == -CUDART_INF_F ? 0.f : sum * ex2_approx(mx - x)) + 1.f;
        mx = x;
      } else if (x != -CUDART_INF_F) {
        sum += ex2_approx(x - mx);
      }
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, mx, off);
      const float s2 = __shfl_xor_sync(0xffffffffu, sum, off);
      const float m = fmaxf(mx, m2);
      if (m != -CUDART_INF_F)
        sum = (mx == -CUDART_INF_F ? 0.f : sum * ex2_approx(mx - m)) +
              (m2 == -CUDART_INF_F ? 0.f : s2 * ex2_approx(m2 - m));
      mx = m;
    }
    const float lse = sum > 0.f ? mx + log2f(sum) : -CUDART_INF_F;
    float acc[kPer];
#pragma unroll
    for (int c = 0; c < kPer; ++c) acc[c] = 0.f;
    const float *sc_r = A.part_scale + s0 * kPairRows + r;
    const uint16_t *o_r = A.part_o + (s0 * kPairRows + r) * HD + lane * kPer;
    for (int k0 = 0; k0 < cnt; k0 += 8) {
      float lk[8], sk[8], v[8][kPer];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        if (k0 + e < cnt) {
          const int64_t off = static_cast<int64_t>(k0 + e) * kPairRows;
          lk[e] = ld_cg_f(lse_r + off);
          sk[e] = ld_cg_f(sc_r + off);
          if constexpr (kPer == 4) {
            const uint2 x = ld_cg_u2(o_r + off * HD);
            const float2 a = half2_to_f2(x.x), b = half2_to_f2(x.y);
            v[e][0] = a.x; v[e][1] = a.y; v[e][2] = b.x; v[e][3] = b.y;
          } else {
            const float2 a = half2_to_f2(ld_cg_u1(o_r + off * HD));
            v[e][0] = a.x; v[e][1] = a.y;
          }
        }
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        if (k0 + e < cnt) {
          const float w = lse == -CUDART_INF_F ? 0.f : ex2_approx(lk[e] - lse) * sk[e];
#pragma unroll
          for (int c = 0; c < kPer; ++c) acc[c] = fmaf(w, v[e][c], acc[c]);
        }
      }
    }
    const int hq_idx = seg.head * A.group + rr % A.group;
    uint16_t *dst = A.out + (t * A.hq + hq_idx) * HD + lane * kPer;
    if constexpr (kPer == 4)
      *reinterpret_cast<uint2 *>(dst) = make_uint2(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]));
    else
      *reinterpret_cast<uint32_t *>(dst) = pack_bf16x2(acc[0], acc[1]);
    if (lane == 0 && A.lse) A.lse[static_cast<int64_t>(hq_idx) * A.n + t] = lse * 0.69314718055994531f;
  }
  return true;
}

template <int HD>
__device__ __noinline__ void step_merge_shares(const StepParams &p, int T, int w8, int lane, volatile int *abort) {
  StepWalker walk = make_walker(p);
  Seg seg;
  while (walk.next(p, T, seg))
    if (seg.merges > 0 && (seg.share >> 8) > 1)
      if (!step_merge_share<HD>(p, seg, T, w8, lane, abort)) return;
}

// ============================================================ the kernel
template <int HD, bool kStep>
__global__ void __launch_bounds__(kPairThreads, 1)
    attn_pair_kernel(const __grid_constant__ typename PairTraits<kStep>::Params p) {
  using C = PairCfg<HD>;
  const AttnParams &A = attn_of(p);
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  PairBars *bars = reinterpret_cast<PairBars *>(smem + C::kBarOff);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int T = kBM / A.group;

  if (threadIdx.x == 0) {
    // fused form: the eight softmax warps write the Q tiles (one arrival each)
    mbar_init(&bars->q_full, kStep ? 8 : 1);
    mbar_init(&bars->q_empty, 1);
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], 1);
      mbar_init(&bars->v_full[s], 1);
      mbar_init(&bars->v_empty[s], 1);
    }
    for (int w = 0; w < 2; ++w) {
      mbar_init(&bars->s_full[w], 1);
      mbar_init(&bars->p_full[w], 4);   // one arrival per softmax warp
      mbar_init(&bars->o_final[w], 1);
      mbar_init(&bars->o_free[w], 4);
    }
    mbar_init(&bars->drain, 1);
    mbar_init(&bars->qraw_full, 1);
    bars->abort = 0;
    fence_barrier_init();
  }
  if (warp == 8 && lane == 0) {
    if constexpr (!kStep) tma_prefetch_desc(&A.tm_q);
    if constexpr (kStep) tma_prefetch_desc(&p.tm_qraw);
    tma_prefetch_desc(&A.tm_k);
    tma_prefetch_desc(&A.tm_v);
  }
  if (warp == 9) {
    tmem_alloc(&bars->tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  TurnSplit *turns = reinterpret_cast<TurnSplit *>(smem + C::kTurnOff);
  int32_t *ids_s = reinterpret_cast<int32_t *>(smem + C::kIdsOff);
  if constexpr (kStep) {
    // RoPE frequencies and the new page ids into shared memory (lanes read
    // them at different indices; parameter reads would serialise)
    if (threadIdx.x < HD / 2) turns[threadIdx.x] = p.inv_turns[threadIdx.x];
    for (int i = threadIdx.x; i < min(p.n_ids, C::kSmemIds); i += kPairThreads) ids_s[i] = p.ids[i];
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // Fused form: the cache, the page table and the partial buffers may still
  // be read or written by the previous kernel, so every role waits for it
  // before its first access to them (the softmax warps first rotate their
  // first queries, inputs of this call).  Item form: the previous kernel is
  // K1, which lets this grid start only once every earlier kernel of the
  // stream has completed; K1 itself writes the packed queries, the keys and
  // values at positions >= L and the page-table entries of the new pages.
  // The MMA warp waits for K1 and issues the first item's queries; the
  // producer stages page ids and loads cached K/V tiles meanwhile, and waits
  // for K1 only before a block that reaches position L.  The partial and
  // output buffers were last read by kernels that completed before K1 started.
  const uint32_t tmem = bars->tmem_base;
  volatile int *abort = &bars->abort;
  auto walk = make_walker(p);
  Seg seg;

  if (warp == 8) {
    // ------------------------------------------------------ TMA producer
    // The whole warp runs the loop (as the MMA issuer does); the elected lane's
    // predicate gates the expect-tx arrivals and the TMA issues.
    int32_t *stage = reinterpret_cast<int32_t *>(smem + C::kPtOff);
    const int ppt = kBN / A.page_size;
    const int tiles_per_block = C::kPtStage / ppt;
    const uint32_t leader = elect_lane();
    uint32_t q_round = 0, k_it = 0, v_it = 0;
    bool ok = true;
    bool appended = false;   // fused form: the launch's new keys are in the cache
    bool pending = false;
    bool waited = kStep;     // item form: K1 has completed (griddepcontrol.wait passed)
    auto await_k1 = [&] {
      if (!waited) {
        pdl_wait();
        waited = true;
      }
    };
    if constexpr (kStep) {
      // the first piece's raw queries before waiting for the previous kernel
      // (they are inputs of this call); then every cache access waits
      pending = walk.next(p, T, seg);
      if (pending) {
        step_qraw_issue<HD>(leader, p, smem, &bars->qraw_full, seg.head, seg.pair, T);
        q_round = 1;
      }
      pdl_wait();
    }
    while (ok && (pending || walk.next(p, T, seg))) {
      if constexpr (kStep) {
        if (!pending) {
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_empty, (q_round - 1) & 1, abort, A.err,
                                                 CSR_DEVERR_WAIT_TIMEOUT));
          if (!ok) break;
          step_qraw_issue<HD>(leader, p, smem, &bars->qraw_full, seg.head, seg.pair, T);
          ++q_round;
        }
        pending = false;
      } else {
        // the first item's queries are issued by the MMA warp once K1 is done
        if (q_round > 0) {
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_empty, (q_round - 1) & 1, abort, A.err,
                                                 CSR_DEVERR_WAIT_TIMEOUT));
          if (!ok) break;
          await_k1();
          item_q_issue<HD>(leader, A, smem, &bars->q_full, seg);
        }
        ++q_round;
      }
      for (int64_t jb = seg.j0; ok && jb < seg.j1; jb += tiles_per_block) {
        const int64_t je = min(jb + tiles_per_block, seg.j1);
        const int npages = static_cast<int>(je - jb) * ppt;
        // item form: a block reaching position L stages page ids K1 may write
        if constexpr (!kStep)
          if (je * kBN > A.L) await_k1();
        __syncwarp();
        // every lane's page-table loads are issued before any is used (one
        // memory round trip per block instead of one per 32 pages)
        constexpr int kPer = C::kPtStage / 32;
        int32_t phys_v[kPer];
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
          const int i = lane + 32 * q;
          const int64_t lp = jb * ppt + i;
          phys_v[q] = 0;
          if (i < npages) {
            if constexpr (kStep) {
              // the launch's new pages come from its id list: staging never
              // waits for the append, only the TMA of the new keys does
              phys_v[q] = (lp < A.n_pages_valid) ? step_page(p, ids_s, lp) : A.page_table[0];
            } else {
              phys_v[q] = (lp < A.n_pages_valid) ? A.page_table[lp] : A.page_table[0];
            }
          }
        }
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
          const int i = lane + 32 * q;
          if (i < npages) {
            int32_t phys = phys_v[q];
            if (phys < 0 || phys >= A.pool_pages) {
              atomicOr(A.err, CSR_DEVERR_BAD_PAGE);
              phys = 0;
            }
            stage[i] = phys;
          }
        }
        __syncwarp();
        for (int64_t j = jb; j < je; ++j) {
          if constexpr (kStep) {
            // key tiles at or past the page holding position L hold the new keys
            if (!appended && (j + 1) * ppt > p.new_lp) {
              if (lane == 0) ok = wait_counter(p.sync, p.append_target, A.err, abort);
              ok = __shfl_sync(0xffffffffu, ok, 0);
              if (!ok) break;
              fence_proxy_async_global();
              appended = true;
            }
          }
          const int32_t *phys = stage + static_cast<int>(j - jb) * ppt;
          const int ks = k_it % C::kStages;
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->k_empty[ks], ((k_it / C::kStages) & 1) ^ 1,
                                                 abort, A.err, CSR_DEVERR_WAIT_TIMEOUT));
          if (!ok) break;
          mbar_arrive_expect_tx_if(leader, &bars->k_full[ks], C::kTileBytes);
          load_kv_tile_if<HD>(leader, A, &A.tm_k, smem + C::kKOff + ks * C::kTileBytes,
                              &bars->k_full[ks], seg.head, phys);
          ++k_it;
          const int vs = v_it % C::kStages;
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->v_empty[vs], ((v_it / C::kStages) & 1) ^ 1,
                                                 abort, A.err, CSR_DEVERR_WAIT_TIMEOUT));
          if (!ok) break;
          mbar_arrive_expect_tx_if(leader, &bars->v_full[vs], C::kTileBytes);
          load_kv_tile_if<HD>(leader, A, &A.tm_v, smem + C::kVOff + vs * C::kTileBytes,
                              &bars->v_full[vs], seg.head, phys);
          ++v_it;
        }
      }
    }
    // every CTA of the item form waits for K1 before it completes, so that a
    // kernel after this one that waits for it also waits for K1
    if constexpr (!kStep) await_k1();
    if (!ok && lane == 0) {
      if (q_round > 0) drain_wait(kStep ? &bars->qraw_full : &bars->q_full, (q_round - 1) & 1);
      for (uint32_t i = (k_it > C::kStages ? k_it - C::kStages : 0); i < k_it; ++i)
        drain_wait(&bars->k_full[i % C::kStages], (i / C::kStages) & 1);
      for (uint32_t i = (v_it > C::kStages ? v_it - C::kStages : 0); i < v_it; ++i)
        drain_wait(&bars->v_full[i % C::kStages], (i / C::kStages) & 1);
    }
  } else if (warp == 9) {
    // ------------------------------------------------------ MMA issuer
    // The whole warp runs the issue loop (operands are warp-uniform) and an
    // elected lane issues each MMA and commit.
    constexpr uint32_t idesc_s = idesc_bf16_f32(kBM, kBN, false, false);
    constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, HD, false, true);
    const uint64_t q_desc = sdesc_sw128(smem_u32(smem + C::kQOff), 16, 1024);
    const uint64_t k_desc = sdesc_sw128(smem_u32(smem + C::kKOff), 16, 1024);
    const uint64_t v_desc = sdesc_sw128(smem_u32(smem + C::kVOff), kBN * 128, 1024);
    uint32_t q_round = 0, k_it = 0, v_it = 0, seg_n = 0;
    uint32_t pv_n[2] = {0, 0};
    bool ok = true;
    if constexpr (kStep) {
      pdl_wait();
    } else {
      // Item form: the first item's queries as soon as K1 is done (they are
      // K1's output); the producer meanwhile stages page ids and the first
      // cached K/V tiles.
      PairWalker first{static_cast<int32_t>(blockIdx.x)};
      Seg s0;
      if (first.next(A, T, s0)) {
        pdl_wait();
        item_q_issue<HD>(elect_lane(), A, smem, &bars->q_full, s0);
      }
    }
    auto wait = [&](uint64_t *bar, uint32_t parity) {
      if (ok)
        ok = __all_sync(0xffffffffu, mbar_wait(bar, parity, abort, A.err, CSR_DEVERR_WAIT_TIMEOUT));
      return ok;
    };
    // S_X = Q_X K^T for tile x from K stage ks
    auto issue_s = [&](int x, int ks) {
      const uint64_t qx = sdesc_advance(q_desc, x * C::kQBytes);
      const uint64_t kst = sdesc_advance(k_desc, ks * C::kTileBytes);
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const uint32_t off = (kk >> 2) * (kBM * 128) + (kk & 3) * 32;
        mma_bf16_ss_warp(tmem + x * kBN, sdesc_advance(qx, off),
                         sdesc_advance(kst, (kk >> 2) * (kBN * 128) + (kk & 3) * 32), idesc_s,
                         kk > 0 ? 1u : 0u);
      }
      mma_commit_warp(&bars->s_full[x]);
    };
    // O_X += P_X V for tile x from V stage vs
    auto issue_pv = [&](int x, int vs, bool first) {
      const uint64_t vst = sdesc_advance(v_desc, vs * C::kTileBytes);
#pragma unroll
      for (int kk = 0; kk < kBN / 16; ++kk)
        mma_bf16_ts_warp(tmem + C::kOCol + x * HD, tmem + x * kBN + kk * 8,
                         sdesc_advance(vst, kk * (16 * 128)), idesc_pv,
                         (!first || kk > 0) ? 1u : 0u);
    };
    while (ok && walk.next(p, T, seg)) {
      if (!wait(&bars->q_full, q_round & 1)) break;
      ++q_round;
      tc_fence_after();
      const int nj = static_cast<int>(seg.j1 - seg.j0);
      int ks = k_it % C::kStages;
      if (!wait(&bars->k_full[ks], (k_it / C::kStages) & 1)) break;
      tc_fence_after();
      issue_s(0, ks);
      issue_s(1, ks);
      mma_commit_warp(&bars->k_empty[ks]);
      ++k_it;
      if (nj == 1) mma_commit_warp(&bars->q_empty);
      for (int i = 0; i < nj; ++i) {
        const int vs = v_it % C::kStages;
        const bool more = i + 1 < nj;
        // ---- tile A
        if (!wait(&bars->p_full[0], pv_n[0] & 1)) break;
        if (!wait(&bars->v_full[vs], (v_it / C::kStages) & 1)) break;
        if (i == 0 && seg_n > 0 && !wait(&bars->o_free[0], (seg_n & 1) ^ 1)) break;
        tc_fence_after();
        issue_pv(0, vs, i == 0);
        if (i == nj - 1) mma_commit_warp(&bars->o_final[0]);
        ++pv_n[0];
        if (more) {
          ks = k_it % C::kStages;
          if (!wait(&bars->k_full[ks], (k_it / C::kStages) & 1)) break;
          tc_fence_after();
          issue_s(0, ks);
        }
        // ---- tile B
        if (!wait(&bars->p_full[1], pv_n[1] & 1)) break;
        if (i == 0 && seg_n > 0 && !wait(&bars->o_free[1], (seg_n & 1) ^ 1)) break;
        tc_fence_after();
        issue_pv(1, vs, i == 0);
        if (i == nj - 1) mma_commit_warp(&bars->o_final[1]);
        ++pv_n[1];
        mma_commit_warp(&bars->v_empty[vs]);
        ++v_it;
        if (more) {
          issue_s(1, ks);
          mma_commit_warp(&bars->k_empty[ks]);
          ++k_it;
          if (i + 1 == nj - 1) mma_commit_warp(&bars->q_empty);
        }
      }
      ++seg_n;
    }
    if (!ok) {
      mma_commit_warp(&bars->drain);
      drain_wait(&bars->drain, 0);
    }
  } else {
    // ------------------------------------------------------ softmax warpgroups
    const int wg = warp >> 2;                  // 0: tile A, 1: tile B
    const int row = threadIdx.x - wg * 128;    // TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t s_col = wg * kBN;
    const uint32_t o_col = C::kOCol + wg * HD;
    uint32_t s_it = 0, seg_n = 0;
    bool ok = true;
    bool pending = false;   // fused form: the first piece, taken before the loop
    uint8_t *qtile = smem + C::kQOff + wg * C::kQBytes;
    float2 *ang = reinterpret_cast<float2 *>(smem + C::kAngOff) + warp * C::kAngEntries;
    if constexpr (kStep) {
      // the first piece's queries before waiting for the previous kernel
      pending = walk.next(p, T, seg);
      if (pending && !step_q_prep<HD>(p, qtile, ang, turns, &bars->qraw_full, 0, &bars->q_full, abort,
                                      seg.pair, wg, row, lane, T))
        ok = false;
      pdl_wait();
      // this CTA's share of the new keys/values, then one arrival per CTA
      // (every softmax thread gets here exactly once)
      step_append<HD>(p, turns, ids_s, threadIdx.x, 256);
      named_sync(3, 256);
      if (threadIdx.x == 0) {
        __threadfence();
        red_release_gpu_add(p.sync, 1u);
      }
    }
    while (ok && (pending || walk.next(p, T, seg))) {
      pending = false;
      if constexpr (kStep) {
        if (seg_n > 0) {
          // the unit's queries, rotated in place once the producer's raw copy
          // (issued after the previous piece's last score MMA) is in
          if (!step_q_prep<HD>(p, qtile, ang, turns, &bars->qraw_full, seg_n & 1, &bars->q_full, abort,
                               seg.pair, wg, row, lane, T)) {
            ok = false;
            break;
          }
        }
      }
      const int tile = seg.pair * 2 + wg;
      const int64_t t = static_cast<int64_t>(tile) * T + row / A.group;
      const bool valid = tile < A.n_tiles && t < A.n;
      const int64_t limit = valid ? A.L + t : -1;
      float m_ref = -CUDART_INF_F;
      float l = 0.f;
      const int nj = static_cast<int>(seg.j1 - seg.j0);
      for (int i = 0; i < nj; ++i) {
        const int64_t j = seg.j0 + i;
        const bool got = mbar_wait(&bars->s_full[wg], s_it & 1, abort, A.err,
                                   CSR_DEVERR_WAIT_TIMEOUT);
        if (!__all_sync(0xffffffffu, got)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // The scores and their row maximum in one load (the TMEM load path
        // reduces); tiles that reach past the row's causal limit mask the
        // later keys and take the maximum of what is left.
        uint32_t sr[kBN];
        float mx = tmem_ld128_rowmax_wait(tmem + lane_base + s_col, sr);
        float s[kBN];
#pragma unroll
        for (int c = 0; c < kBN; ++c) s[c] = __uint_as_float(sr[c]);
        const int64_t key0 = j * kBN;
        if (key0 + kBN - 1 > limit) {
#pragma unroll
          for (int c = 0; c < kBN; ++c)
            if (key0 + c > limit) s[c] = -CUDART_INF_F;
          // three operands per instruction, eight independent chains
          float mp[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) mp[e] = fmaxf(s[2 * e], s[2 * e + 1]);
#pragma unroll
          for (int c = 16; c < kBN; c += 2) mp[(c >> 1) & 7] = max3f(mp[(c >> 1) & 7], s[c], s[c + 1]);
          mx = max3f(max3f(mp[0], mp[1], mp[2]), max3f(mp[3], mp[4], mp[5]), fmaxf(mp[6], mp[7]));
        }
        const float mx_s = mx * A.scale_log2;
        const bool need = mx_s > m_ref + 8.0f;
        const float m_new = need ? mx_s : m_ref;
        const float alpha = need ? ex2_approx(m_ref - m_new) : 1.0f;
        const bool had_mass = l > 0.f;
        l *= alpha;
        m_ref = m_new;
        const float m_use = (m_ref == -CUDART_INF_F) ? 0.f : m_ref;
        // p = 2^(s * scale_log2 - m): the scale-and-shift and the row sum run
        // on packed fp32 pairs, the exponentials one lane at a time.
        const uint64_t scale2 = f32x2(A.scale_log2, A.scale_log2);
        const uint64_t shift2 = f32x2(-m_use, -m_use);
        uint64_t rp2[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) rp2[e] = 0ull;  // (+0.0f, +0.0f)
        uint32_t pk[kBN / 2];
#pragma unroll
        for (int c = 0; c < kBN; c += 2) {
          float x0, x1;
          f32x2_split(fma_f32x2(f32x2(s[c], s[c + 1]), scale2, shift2), x0, x1);
          const float p0 = ex2_approx(x0);
          const float p1 = ex2_approx(x1);
          rp2[(c >> 1) & 3] = add_f32x2(rp2[(c >> 1) & 3], f32x2(p0, p1));
          pk[c / 2] = pack_bf16x2(p0, p1);
        }
        float r[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) f32x2_split(rp2[e], r[2 * e], r[2 * e + 1]);
        l += ((r[0] + r[1]) + (r[2] + r[3])) + ((r[4] + r[5]) + (r[6] + r[7]));
        tmem_st64(tmem + lane_base + s_col, pk);
        // PV of the previous tile finished before these scores were published
        // (same commit), so O can be rescaled here without another wait.
        if (i > 0 && __any_sync(0xffffffffu, need && had_mass))
          rescale_o<HD>(tmem + lane_base + o_col, alpha);
        tmem_st_wait();
        tc_fence_before();
        // One arrival per warp once all its lanes have stored P: 128 arrivals
        // on one barrier serialise in shared memory (measured 3.5% slower).
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->p_full[wg]);
        ++s_it;
      }
      if (!ok) break;
      // ---------------------------------------------------- epilogue
      const bool got_o = mbar_wait(&bars->o_final[wg], seg_n & 1, abort, A.err,
                                   CSR_DEVERR_WAIT_TIMEOUT);
      if (!__all_sync(0xffffffffu, got_o)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float inv_l = l > 0.f ? 1.0f / l : 0.f;
      float lse2 = l > 0.f ? m_ref + log2f(l) : -CUDART_INF_F;
      uint32_t o[HD];
      load_o<HD>(tmem + lane_base + o_col, o);
      // O is in registers now: the MMA warp may accumulate the next piece
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->o_free[wg]);
      bool to_out = seg.complete;
      if constexpr (kStep) {
        if (seg.merges > 0 && (seg.share >> 8) <= 1) {
          // The unit's last piece: once the other pieces have written this
          // warp's rows (their flags hold this launch's generation), combine
          // lse = log2(2^lse_own + sum_k 2^lse_k) and
          // out = 2^(lse_own - lse) O_own / l + sum_k 2^(lse_k - lse) O_k.
          const uint32_t *fl = p.flags + static_cast<int64_t>(seg.slot) * 8 + warp;
          bool got = true;
          for (int k = 0; k < seg.merges && got; ++k) got = wait_counter(fl + k * 8, p.gen, A.err, abort);
          if (!__all_sync(0xffffffffu, got)) {
            ok = false;
            break;
          }
          const int64_t r0 = static_cast<int64_t>(seg.slot) * kPairRows + wg * kBM + row;
          float mx = lse2;
          for (int k = 0; k < seg.merges; ++k) mx = fmaxf(mx, ld_cg_f(A.part_lse + r0 + k * kPairRows));
          const float m_use = mx == -CUDART_INF_F ? 0.f : mx;
          float sum = l > 0.f ? ex2_approx(lse2 - m_use) : 0.f;
          for (int k = 0; k < seg.merges; ++k) sum += ex2_approx(ld_cg_f(A.part_lse + r0 + k * kPairRows) - m_use);
          const float lse_t = sum > 0.f ? m_use + log2f(sum) : -CUDART_INF_F;
          const float w_own = l > 0.f ? ex2_approx(lse2 - lse_t) * inv_l : 0.f;
#pragma unroll
          for (int c = 0; c < HD; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * w_own);
          for (int k = 0; k < seg.merges; ++k) {
            const int64_t rk = r0 + k * kPairRows;
            const float lk = ld_cg_f(A.part_lse + rk);
            const float wk = lse_t == -CUDART_INF_F ? 0.f : ex2_approx(lk - lse_t) * ld_cg_f(A.part_scale + rk);
            const uint16_t *src = A.part_o + rk * HD;
#pragma unroll
            for (int c0 = 0; c0 < HD; c0 += 32) {
              uint4 v[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) v[e] = ld_cg_u4(src + c0 + 8 * e);
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const uint32_t q[4] = {v[e].x, v[e].y, v[e].z, v[e].w};
#pragma unroll
                for (int h = 0; h < 4; ++h) {
                  const float2 f = half2_to_f2(q[h]);
                  const int c = c0 + 8 * e + 2 * h;
                  o[c] = __float_as_uint(fmaf(wk, f.x, __uint_as_float(o[c])));
                  o[c + 1] = __float_as_uint(fmaf(wk, f.y, __uint_as_float(o[c + 1])));
                }
              }
            }
          }
          inv_l = 1.0f;
          lse2 = lse_t;
          to_out = true;
        }
      }
      if (to_out) {
        if (valid) {
          const int hq_idx = seg.head * A.group + row % A.group;
          uint16_t *dst = A.out + (static_cast<int64_t>(t) * A.hq + hq_idx) * HD;
#pragma unroll
          for (int q8 = 0; q8 < HD / 8; ++q8) {
            uint32_t w[4];
#pragma unroll
            for (int c = 0; c < 4; ++c)
              w[c] = pack_bf16x2(__uint_as_float(o[q8 * 8 + 2 * c]) * inv_l,
                                 __uint_as_float(o[q8 * 8 + 2 * c + 1]) * inv_l);
            reinterpret_cast<uint4 *>(dst)[q8] = make_uint4(w[0], w[1], w[2], w[3]);
          }
          if (A.lse) A.lse[static_cast<int64_t>(hq_idx) * A.n + t] = lse2 * 0.69314718055994531f;
        }
      } else {
        const int64_t base = static_cast<int64_t>(seg.slot) * kPairRows + wg * kBM + row;
        // the row scaled by its largest magnitude, in fp16 (the partial
        // buffer is 256-byte aligned and rows are HD halves: 32-byte stores)
        float mx = 0.f;
#pragma unroll
        for (int c = 0; c < HD; ++c) mx = fmaxf(mx, fabsf(__uint_as_float(o[c])));
        const float inv_s = mx > 0.f ? 1.0f / mx : 0.f;
        uint16_t *dst = A.part_o + base * HD;
#pragma unroll
        for (int c = 0; c < HD / 16; ++c) {
          uint32_t w[8];
#pragma unroll
          for (int e = 0; e < 8; ++e)
            w[e] = f2_to_half2(__uint_as_float(o[16 * c + 2 * e]) * inv_s, __uint_as_float(o[16 * c + 2 * e + 1]) * inv_s);
          st_global_v8(dst + 16 * c, w);
        }
        A.part_scale[base] = mx * inv_l;
        A.part_lse[base] = lse2;
        if constexpr (kStep) {
          // this warp's 32 rows are written: raise the slot's flag for the
          // unit's last piece
          __threadfence();
          __syncwarp();
          if (lane == 0) st_release_gpu(p.flags + static_cast<int64_t>(seg.slot) * 8 + warp, p.gen);
          // a member of a last group of several pieces merges its share
          // after this CTA's last piece
        }
      }
      ++seg_n;
    }
    if constexpr (kStep) {
      // The merge shares of this CTA's pieces in larger last groups (every
      // flag of this CTA is raised by now, so these waits hold up no one).
      if (ok) step_merge_shares<HD>(p, T, warp, lane, abort);
    }
  }

  pdl_launch_dependents();
  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ------------------------------------------------------------------ K3 merge
// 16-byte global loads of eight fp16 values (the partial buffer is 256-byte
// aligned and its rows are HD halves, so every lane's eight start on a
// 16-byte boundary), converted when used.
__device__ __forceinline__ uint4 ld_global_u4(const void *ptr) {
  uint4 v;
  asm volatile("ld.global.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(ptr));
  return v;
}
// acc += w * (the eight fp16 values in q)
__device__ __forceinline__ void fma_half8(float (&acc)[8], float w, const uint4 &q) {
  const uint32_t h[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = half2_to_f2(h[i]);
    acc[2 * i] = fmaf(w, f.x, acc[2 * i]);
    acc[2 * i + 1] = fmaf(w, f.y, acc[2 * i + 1]);
  }
}

// K3: combine the split-KV partials of every row: lse = log2(sum_k 2^lse_k),
// out = sum_k 2^(lse_k - lse) * s_k * O'_k (O_k = s_k O'_k, normalised by its
// own row sum, stored as fp16 O'_k with its scale s_k).  A row is read by a
// group of HD / 8 lanes (eight values, one 16-byte load per lane per chunk);
// a block of 256 threads holds 256 / (HD/8)
// such slots.  The merge is bound by how many bytes are in flight, so every
// load of a slot -- the LSEs of all chunks and up to kMergeChunksPerSlot
// partial rows -- is issued before any is used; rows with more chunks are
// spread over p.slots_per_row slots whose shares are summed in shared memory.
// Rows with more than 64 chunks loop over their chunks.
template <int HD>
__global__ void __launch_bounds__(256, 4) merge_kernel(const __grid_constant__ MergeParams p) {
  constexpr int kLanes = HD / 8;            // lanes per slot (16 or 8)
  constexpr int kSlots = 256 / kLanes;      // slots per block (16 or 32)
  constexpr int kLse = 64 / kLanes;         // LSE registers per lane for up to 64 chunks
  constexpr int kC = kMergeChunksPerSlot;
  __shared__ float red[kSlots][HD];
  pdl_wait();   // the partials come from the attention kernel
  const int head = blockIdx.x / p.n_tiles;
  const int tile = blockIdx.x - head * p.n_tiles;
  const int T = kBM / p.group;
  const int uph = (p.n_tiles + 1) / 2;      // pairs per head
  const int pair = tile / 2;
  const int half = tile - pair * 2;
  const int64_t kv = unit_iters(p.L, p.n, T, pair * 2 + 1);
  const int nk = static_cast<int>((kv + p.chunk_tiles - 1) / p.chunk_tiles);
  if (nk <= 1) return;  // the whole block: written whole by the attention kernel
  const int spr = p.slots_per_row;
  const int slot = threadIdx.x / kLanes;
  const int sl = threadIdx.x % kLanes;
  const int sub = slot % spr;
  const int r = blockIdx.y * (kSlots / spr) + slot / spr;
  const int64_t t = static_cast<int64_t>(tile) * T + r / p.group;
  const bool valid = r < kBM && t < p.n;
  const int64_t units = static_cast<int64_t>(p.hkv) * uph;
  const int64_t row_in_item = static_cast<int64_t>(half) * kBM + r;
  // row index (item * kPairRows + row_in_item) of chunk k's partial
  auto prow = [&](int k) {
    return (static_cast<int64_t>(k) * units + static_cast<int64_t>(head) * uph + pair) * kPairRows +
           row_in_item;
  };
  float acc[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) acc[e] = 0.f;
  float lse2 = -CUDART_INF_F;
  // Shuffles run on every lane (rows past n included) and stay within a slot.
  auto slot_max = [&](float x) {
#pragma unroll
    for (int off = kLanes / 2; off > 0; off >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, off, kLanes));
    return x;
  };
  auto slot_sum = [&](float x) {
#pragma unroll
    for (int off = kLanes / 2; off > 0; off >>= 1) x += __shfl_xor_sync(0xffffffffu, x, off, kLanes);
    return x;
  };
  if (nk <= 64 && nk <= kC * spr) {
    // lane sl holds the LSEs of chunks sl, sl + kLanes, ...
    float l[kLse];
#pragma unroll
    for (int i = 0; i < kLse; ++i) {
      const int k = sl + i * kLanes;
      l[i] = (valid && k < nk) ? p.part_lse[prow(k)] : -CUDART_INF_F;
    }
    // this slot's chunks: their partial rows and (the same address on every
    // lane of the slot) their LSEs
    uint4 v[kC];
    float lk[kC], sk[kC];
#pragma unroll
    for (int u = 0; u < kC; ++u) {
      const int k = sub + u * spr;
      if (valid && k < nk) {
        lk[u] = p.part_lse[prow(k)];
        sk[u] = p.part_scale[prow(k)];
        v[u] = ld_global_u4(p.part_o + prow(k) * HD + sl * 8);
      } else {
        lk[u] = -CUDART_INF_F;
        sk[u] = 0.f;
        v[u] = make_uint4(0u, 0u, 0u, 0u);
      }
    }
    float mx = l[0];
#pragma unroll
    for (int i = 1; i < kLse; ++i) mx = fmaxf(mx, l[i]);
    mx = slot_max(mx);
    const float m_use = mx == -CUDART_INF_F ? 0.f : mx;
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < kLse; ++i) sum += ex2_approx(l[i] - m_use);   // 0 for absent chunks
    sum = slot_sum(sum);
    lse2 = sum > 0.f ? m_use + log2f(sum) : -CUDART_INF_F;
    if (sum > 0.f) {
#pragma unroll
      for (int u = 0; u < kC; ++u) fma_half8(acc, ex2_approx(lk[u] - lse2) * sk[u], v[u]);
    }
  } else {
    float mx = -CUDART_INF_F;
    for (int k = sl; k < nk; k += kLanes) mx = fmaxf(mx, valid ? p.part_lse[prow(k)] : -CUDART_INF_F);
    mx = slot_max(mx);
    const float m_use = mx == -CUDART_INF_F ? 0.f : mx;
    float sum = 0.f;
    for (int k = sl; k < nk; k += kLanes) sum += valid ? ex2_approx(p.part_lse[prow(k)] - m_use) : 0.f;
    sum = slot_sum(sum);
    lse2 = sum > 0.f ? m_use + log2f(sum) : -CUDART_INF_F;
    if (valid && sum > 0.f) {
      for (int k = sub; k < nk; k += spr) {
        const int64_t base = prow(k);
        const float w = ex2_approx(p.part_lse[base] - lse2) * p.part_scale[base];
        fma_half8(acc, w, ld_global_u4(p.part_o + base * HD + sl * 8));
      }
    }
  }
  if (spr > 1) {   // sum the row's shares
#pragma unroll
    for (int x = 0; x < 8; ++x) red[slot][sl * 8 + x] = acc[x];
    __syncthreads();
    if (sub == 0) {
      for (int w = 1; w < spr; ++w)
#pragma unroll
        for (int x = 0; x < 8; ++x) acc[x] += red[slot + w][sl * 8 + x];
    }
  }
  if (!valid || sub != 0) return;
  const int hq_idx = head * p.group + r % p.group;
  uint16_t *dst = p.out + (t * p.hq + hq_idx) * HD + sl * 8;
  *reinterpret_cast<uint4 *>(dst) = make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]),
                                               pack_bf16x2(acc[4], acc[5]), pack_bf16x2(acc[6], acc[7]));
  if (sl == 0 && p.lse) p.lse[static_cast<int64_t>(hq_idx) * p.n + t] = lse2 * 0.69314718055994531f;
}

cudaError_t attn_configure(int head_dim) {
  const auto attr = cudaFuncAttributeMaxDynamicSharedMemorySize;
  cudaError_t e;
  if (head_dim == 64) {
    e = cudaFuncSetAttribute(attn_pair_kernel<64, false>, attr, PairCfg<64>::kSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(attn_pair_kernel<64, true>, attr, PairCfg<64>::kSmemStep);
  } else {
    e = cudaFuncSetAttribute(attn_pair_kernel<128, false>, attr, PairCfg<128>::kSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(attn_pair_kernel<128, true>, attr, PairCfg<128>::kSmemStep);
  }
  return e;
}

// Launch with programmatic stream serialisation (see pdl_wait); cooperative
// launches also guarantee that every CTA of the grid is resident at once.
template <typename... Args>
cudaError_t launch_pdl(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       bool cooperative, const Args &...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeCooperative;
  attr[1].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = cooperative ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

cudaError_t launch_attention(const AttnParams &p, int head_dim, cudaStream_t s) {
  if (head_dim == 64)
    return launch_pdl(attn_pair_kernel<64, false>, dim3(p.grid), dim3(kPairThreads), PairCfg<64>::kSmem, s,
                      false, p);
  return launch_pdl(attn_pair_kernel<128, false>, dim3(p.grid), dim3(kPairThreads), PairCfg<128>::kSmem, s,
                    false, p);
}

cudaError_t launch_step(const StepParams &p, int head_dim, cudaStream_t s) {
  if (head_dim == 64)
    return launch_pdl(attn_pair_kernel<64, true>, dim3(p.s.grid), dim3(kPairThreads), PairCfg<64>::kSmemStep,
                      s, true, p);
  return launch_pdl(attn_pair_kernel<128, true>, dim3(p.s.grid), dim3(kPairThreads), PairCfg<128>::kSmemStep,
                    s, true, p);
}

cudaError_t launch_merge(const MergeParams &p, cudaStream_t s) {
  const int slots = 256 / (p.d / 8);
  const dim3 grid(p.hkv * p.n_tiles, kBM * p.slots_per_row / slots);
  if (p.d == 64) return launch_pdl(merge_kernel<64>, grid, dim3(256), 0, s, false, p);
  return launch_pdl(merge_kernel<128>, grid, dim3(256), 0, s, false, p);
}

}  // namespace csr
