// kernels_attn.cu -- causal attention of a block of new tokens over the paged
// cache (Eq. causal_attention_1..3: a_n = softmax(q_n K_{1:n}^T / sqrt(d_k)),
// o_n = a_n V_{1:n}), on the 5th-generation tensor cores of sm_103a.
//
// Work decomposition.  The rotated queries of one KV head are packed as rows
// t*G + g (token t, group member g), so one 128-row tile holds 128/G tokens of
// all G query heads that read the same keys.  A unit is one (kv head, query
// tile); its key range [0, L + last token of the tile] is cut into n_chunks
// chunks of chunk_tiles 128-key tiles.  An item is one (key chunk, unit);
// items are numbered chunk-major, (chunk, head, tile), and CTA c takes items
// c, c + grid, c + 2 grid, ...  The CTAs running at the same time therefore
// work on the same key chunk and read it through L2 instead of each
// streaming the whole cache from HBM.  A unit that fits in one chunk is
// written directly; otherwise each item writes a normalised partial output
// with its log-sum-exp and K3 merges them.
//
// Kernels.  attn_pair_kernel (the default) gives each CTA two consecutive
// query tiles of one KV head, so every K/V tile staged in shared memory feeds
// both; attn_kernel (one query tile per CTA, two score buffers) and
// attn_pipe_kernel (two query tiles, 64-key tiles, two score buffers each) are
// earlier designs kept behind flags.  Roles of the default (320 threads):
//   warp 8    TMA producer: the two Q tiles, then K and V tiles page by page
//             (page ids staged in shared memory), into 128-byte-swizzled
//             shared-memory stages; the whole warp runs the loop and an
//             elected lane issues the copies;
//   warp 9    MMA issuer: S_X = Q_X K^T (both operands in shared memory) and
//             O_X += P_X V (P from TMEM) for X = A, B, ordered PV_A(i),
//             S_A(i+1), PV_B(i), S_B(i+1); the whole warp runs the loop and
//             elect.sync picks the issuing lane;
//   warps 0-7 softmax, one warpgroup per query tile: one thread per query row
//             (its TMEM lane); reads its scores with the row maximum reduced
//             by the TMEM load (tcgen05.ld.red, sm_103a), masks keys past the
//             row's position, keeps a
//             running max with a lazy rescale of O (only when the max grows
//             by more than 2^8), writes P as bf16 over its own score columns,
//             and finally normalises O and stores it.
// The kernels of a call (K1 rope/append, K2 attention, K3 merge) are chained
// by programmatic dependent launch: K1 releases K2 at its entry and K2
// releases K3 at its end; each runs its setup while its predecessor works and
// waits (griddepcontrol) before its first global access.
// Every wait on an mbarrier is bounded (CSR_DEVERR_WAIT_TIMEOUT).
#include <cuda_bf16.h>
#include <math_constants.h>

#include "../../include/csr.h"
#include "internal.h"
#include "ptx.cuh"

namespace csr {

template <int HD>
struct AttnCfg {
  static constexpr int kStages = (HD == 64) ? 4 : 2;
  static constexpr int kBoxes = HD / 64;                 // 64-column (128-byte) boxes per row
  static constexpr int kQBytes = kBM * HD * 2;
  static constexpr int kTileBytes = kBN * HD * 2;
  static constexpr int kQOff = 0;
  static constexpr int kKOff = kQOff + kQBytes;
  static constexpr int kVOff = kKOff + kStages * kTileBytes;
  static constexpr int kBarOff = kVOff + kStages * kTileBytes;
  static constexpr int kPtOff = kBarOff + 1024;          // staged page ids
  static constexpr int kPtStage = 512;                   // entries per staging block
  static constexpr int kSmem = kPtOff + kPtStage * 4 + 1024;  // + alignment slack
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kOCol = 2 * kBN;             // O accumulator after two S buffers
};

struct Bars {
  uint64_t q_full, q_empty;
  uint64_t k_full[4], k_empty[4], v_full[4], v_empty[4];
  uint64_t s_full[2], s_free[2], p_full[2];
  uint64_t o_done, o_final, o_free, drain;
  uint32_t tmem_base;
  int abort;
};

size_t attn_smem_bytes(int head_dim) {
  return head_dim == 64 ? AttnCfg<64>::kSmem : AttnCfg<128>::kSmem;
}

// One item: a run of key tiles [j0, j1) of one unit.
struct Seg {
  int32_t head, tile, item;
  int32_t nk;  // key chunks of the item's unit
  int64_t j0, j1;
  bool complete;
};

// Walks the CTA's items (c, c + grid, ...); every role walks the same list.
struct ItemWalker {
  int32_t item;
  __device__ bool next(const AttnParams &p, int T, Seg &s) {
    const int32_t units = p.hkv * p.n_tiles;
    while (item < p.n_items) {
      const int32_t it = item;
      item += p.grid;
      const int32_t k = it / units;
      const int32_t rem = it - k * units;
      const int32_t head = rem / p.n_tiles;
      const int32_t tile = rem - head * p.n_tiles;
      const int64_t kv = unit_iters(p.L, p.n, T, tile);
      const int64_t j0 = static_cast<int64_t>(k) * p.chunk_tiles;
      if (j0 >= kv) continue;  // this unit has fewer chunks
      s.head = head;
      s.tile = tile;
      s.item = it;
      s.j0 = j0;
      s.j1 = min(j0 + p.chunk_tiles, kv);
      s.complete = kv <= p.chunk_tiles;
      return true;
    }
    return false;
  }
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

// Issue the TMA loads of keys [key0, key0 + bn) of `head` into a 128B-swizzled
// tile (box b of 64 columns at dst + b * bn * 128).  The copies are pieces of
// min(P, 64) rows (the tensor maps' box height); `phys` holds the physical ids
// of logical pages lp_base, lp_base + 1, ...
template <int HD>
__device__ __forceinline__ void load_kv_keys(const AttnParams &p, const CUtensorMap *map,
                                             uint8_t *dst, int bn, uint64_t *bar, int head,
                                             const int32_t *phys, int64_t lp_base, int64_t key0) {
  const int P = p.page_size;
  const int seg = P < 64 ? P : 64;
  for (int r = 0; r < bn; r += seg) {
    const int64_t key = key0 + r;
    const int64_t lp = key / P;
    const int32_t row = (phys[lp - lp_base] * p.hkv + head) * P + static_cast<int32_t>(key - lp * P);
#pragma unroll
    for (int b = 0; b < HD / 64; ++b) tma_load_2d(dst + b * (bn * 128) + r * 128, map, bar, b * 64, row);
  }
}

// Issue the TMA loads of one 128-key tile of `head` whose pages' physical ids
// are phys[0 .. 128/P): one 64-column box per page and column half (two
// 64-row boxes per page when P = 128).
template <int HD>
__device__ __forceinline__ void load_kv_tile(const AttnParams &p, const CUtensorMap *map,
                                             uint8_t *dst, uint64_t *bar, int head,
                                             const int32_t *phys) {
  const int P = p.page_size;
  const int ppt = kBN / P;
  const int seg = P < 64 ? P : 64;
  for (int pp = 0; pp < ppt; ++pp) {
    const int32_t row0 = (phys[pp] * p.hkv + head) * P;
    for (int r = 0; r < P; r += seg) {
#pragma unroll
      for (int b = 0; b < HD / 64; ++b)
        tma_load_2d(dst + b * (kBN * 128) + (pp * P + r) * 128, map, bar, b * 64, row0 + r);
    }
  }
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

// Stage the physical ids of the logical pages covering key tiles [jb, je)
// (tiles of bn keys) into `stage`, one id per page (whole producer warp).
// Returns the first staged logical page.
__device__ __forceinline__ int64_t stage_pages(const AttnParams &p, int32_t *stage, int bn,
                                               int64_t jb, int64_t je, int lane) {
  const int64_t lp0 = jb * bn / p.page_size;
  const int64_t lp1 = (je * bn + p.page_size - 1) / p.page_size;
  for (int64_t lp = lp0 + lane; lp < lp1; lp += 32) {
    int32_t phys = (lp < p.n_pages_valid) ? p.page_table[lp] : p.page_table[0];
    if (phys < 0 || phys >= p.pool_pages) {
      atomicOr(p.err, CSR_DEVERR_BAD_PAGE);
      phys = 0;
    }
    stage[lp - lp0] = phys;
  }
  return lp0;
}

template <int HD>
__global__ void __launch_bounds__(192, 1) attn_kernel(const __grid_constant__ AttnParams p) {
  using C = AttnCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  Bars *bars = reinterpret_cast<Bars *>(smem + C::kBarOff);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int T = kBM / p.group;
  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->q_empty, 1);
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], 1);
      mbar_init(&bars->v_full[s], 1);
      mbar_init(&bars->v_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars->s_full[s], 1);
      mbar_init(&bars->s_free[s], 1);
      mbar_init(&bars->p_full[s], 128);
    }
    mbar_init(&bars->o_done, 1);
    mbar_init(&bars->o_final, 1);
    mbar_init(&bars->o_free, 128);
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    fence_barrier_init();
  }
  if (warp == 4 && lane == 0) {
    tma_prefetch_desc(&p.tm_q);
    tma_prefetch_desc(&p.tm_k);
    tma_prefetch_desc(&p.tm_v);
  }
  if (warp == 5) {
    tmem_alloc(&bars->tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();   // the block's queries, keys and page table come from the previous kernel
  const uint32_t tmem = bars->tmem_base;
  volatile int *abort = &bars->abort;
  ItemWalker walk{static_cast<int32_t>(blockIdx.x)};
  Seg seg;

  if (warp == 4) {
    // ------------------------------------------------------ TMA producer
    // The whole warp stages the page ids of the next tiles into shared memory
    // (coalesced page-table reads off the critical path); lane 0 issues the
    // copies from there.
    int32_t *stage = reinterpret_cast<int32_t *>(smem + C::kPtOff);
    // key tiles whose pages fit one staging block (a tile may end mid-page)
    const int tiles_per_block = (C::kPtStage - 2) * p.page_size / kBN;
    uint32_t q_round = 0, k_it = 0, v_it = 0;
    bool ok = true;
    while (ok && walk.next(p, T, seg)) {
      if (lane == 0) {
        if (q_round > 0 && !mbar_wait(&bars->q_empty, (q_round - 1) & 1, abort, p.err,
                                      CSR_DEVERR_WAIT_TIMEOUT)) {
          ok = false;
        } else {
          mbar_arrive_expect_tx(&bars->q_full, C::kQBytes);
          const int32_t qrow = seg.head * p.rows_cap + seg.tile * kBM;
#pragma unroll
          for (int b = 0; b < C::kBoxes; ++b)
            tma_load_2d(smem + C::kQOff + b * (kBM * 128), &p.tm_q, &bars->q_full, b * 64, qrow);
          ++q_round;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      for (int64_t jb = seg.j0; ok && jb < seg.j1; jb += tiles_per_block) {
        const int64_t je = min(jb + tiles_per_block, seg.j1);
        __syncwarp();
        const int64_t lp_base = stage_pages(p, stage, kBN, jb, je, lane);
        __syncwarp();
        if (lane == 0) {
          for (int64_t j = jb; j < je; ++j) {

            const int ks = k_it % C::kStages;
            if (!mbar_wait(&bars->k_empty[ks], ((k_it / C::kStages) & 1) ^ 1, abort, p.err,
                           CSR_DEVERR_WAIT_TIMEOUT)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&bars->k_full[ks], C::kTileBytes);
            load_kv_keys<HD>(p, &p.tm_k, smem + C::kKOff + ks * C::kTileBytes, kBN, &bars->k_full[ks],
                             seg.head, stage, lp_base, j * kBN);
            ++k_it;
            const int vs = v_it % C::kStages;
            if (!mbar_wait(&bars->v_empty[vs], ((v_it / C::kStages) & 1) ^ 1, abort, p.err,
                           CSR_DEVERR_WAIT_TIMEOUT)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&bars->v_full[vs], C::kTileBytes);
            load_kv_keys<HD>(p, &p.tm_v, smem + C::kVOff + vs * C::kTileBytes, kBN, &bars->v_full[vs],
                             seg.head, stage, lp_base, j * kBN);
            ++v_it;
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
      }
    }
    if (!ok && lane == 0) {
      // Let the copies already issued land before the CTA's memory goes away.
      if (q_round > 0) drain_wait(&bars->q_full, (q_round - 1) & 1);
      for (uint32_t i = (k_it > C::kStages ? k_it - C::kStages : 0); i < k_it; ++i)
        drain_wait(&bars->k_full[i % C::kStages], (i / C::kStages) & 1);
      for (uint32_t i = (v_it > C::kStages ? v_it - C::kStages : 0); i < v_it; ++i)
        drain_wait(&bars->v_full[i % C::kStages], (i / C::kStages) & 1);
    }
  } else if (warp == 5) {
    if (lane == 0) {
      // ------------------------------------------------------ MMA issuer
      constexpr uint32_t idesc_s = idesc_bf16_f32(kBM, kBN, false, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, HD, false, true);
      const uint32_t q_base = smem_u32(smem + C::kQOff);
      const uint32_t k_base = smem_u32(smem + C::kKOff);
      const uint32_t v_base = smem_u32(smem + C::kVOff);
      uint32_t q_round = 0, k_it = 0, v_it = 0, s_it = 0, pv_it = 0, seg_n = 0;
      bool ok = true;
      while (ok && walk.next(p, T, seg)) {
        if (!mbar_wait(&bars->q_full, q_round & 1, abort, p.err, CSR_DEVERR_WAIT_TIMEOUT)) {
          ok = false;
          break;
        }
        ++q_round;
        tc_fence_after();
        const int nj = static_cast<int>(seg.j1 - seg.j0);
        for (int i = 0; i <= nj && ok; ++i) {
          if (i < nj) {
            const uint32_t sb = s_it & 1;
            const int ks = k_it % C::kStages;
            if (!mbar_wait(&bars->s_free[sb], ((s_it >> 1) & 1) ^ 1, abort, p.err,
                           CSR_DEVERR_WAIT_TIMEOUT) ||
                !mbar_wait(&bars->k_full[ks], (k_it / C::kStages) & 1, abort, p.err,
                           CSR_DEVERR_WAIT_TIMEOUT)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t kst = k_base + ks * C::kTileBytes;
#pragma unroll
            for (int kk = 0; kk < HD / 16; ++kk) {
              const uint64_t a =
                  sdesc_sw128(q_base + (kk >> 2) * (kBM * 128) + (kk & 3) * 32, 16, 1024);
              const uint64_t b =
                  sdesc_sw128(kst + (kk >> 2) * (kBN * 128) + (kk & 3) * 32, 16, 1024);
              mma_bf16_ss(tmem + sb * kBN, a, b, idesc_s, kk > 0 ? 1u : 0u);
            }
            mma_commit(&bars->k_empty[ks]);
            mma_commit(&bars->s_full[sb]);
            if (i == nj - 1) mma_commit(&bars->q_empty);
            ++k_it;
            ++s_it;
          }
          if (i >= 1) {
            const uint32_t pb = pv_it & 1;
            const int vs = v_it % C::kStages;
            if (!mbar_wait(&bars->p_full[pb], (pv_it >> 1) & 1, abort, p.err,
                           CSR_DEVERR_WAIT_TIMEOUT) ||
                !mbar_wait(&bars->v_full[vs], (v_it / C::kStages) & 1, abort, p.err,
                           CSR_DEVERR_WAIT_TIMEOUT)) {
              ok = false;
              break;
            }
            if (i == 1 && seg_n > 0 &&
                !mbar_wait(&bars->o_free, (seg_n & 1) ^ 1, abort, p.err,
                           CSR_DEVERR_WAIT_TIMEOUT)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t vst = v_base + vs * C::kTileBytes;
#pragma unroll
            for (int kk = 0; kk < kBN / 16; ++kk) {
              const uint64_t b = sdesc_sw128(vst + kk * (16 * 128), kBN * 128, 1024);
              mma_bf16_ts(tmem + C::kOCol, tmem + pb * kBN + kk * 8, b, idesc_pv,
                          (i > 1 || kk > 0) ? 1u : 0u);
            }
            mma_commit(&bars->v_empty[vs]);
            mma_commit(&bars->s_free[pb]);
            mma_commit(&bars->o_done);
            if (i == nj) mma_commit(&bars->o_final);  // the segment's last PV
            ++v_it;
            ++pv_it;
          }
        }
        ++seg_n;
      }
      if (!ok) {
        // Wait for the MMAs already issued before TMEM is released.
        mma_commit(&bars->drain);
        drain_wait(&bars->drain, 0);
      }
    }
  } else {
    // ------------------------------------------------------ softmax warps 0-3
    const int row = threadIdx.x;  // TMEM lane of this thread
    const uint32_t lane_base = static_cast<uint32_t>(warp * 32) << 16;
    uint32_t s_it = 0, seg_n = 0;
    bool ok = true;
    while (ok && walk.next(p, T, seg)) {
      const int64_t t = static_cast<int64_t>(seg.tile) * T + row / p.group;
      const bool valid = t < p.n;
      const int64_t limit = valid ? p.L + t : -1;  // last visible key index
      float m_ref = -CUDART_INF_F;
      float l = 0.f;
      const int nj = static_cast<int>(seg.j1 - seg.j0);
      for (int i = 0; i < nj; ++i) {
        const int64_t j = seg.j0 + i;
        const uint32_t sb = s_it & 1;
        const bool got = mbar_wait(&bars->s_full[sb], (s_it >> 1) & 1, abort, p.err,
                                   CSR_DEVERR_WAIT_TIMEOUT);
        if (!__all_sync(0xffffffffu, got)) {  // keep the warp converged for tcgen05.ld
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t sr[kBN];
        tmem_ld128_wait(tmem + lane_base + sb * kBN, sr);  // the whole score row, one wait
        float s[kBN];
#pragma unroll
        for (int c = 0; c < kBN; ++c) s[c] = __uint_as_float(sr[c]);
        const int64_t key0 = j * kBN;
        if (key0 + kBN - 1 > limit) {
#pragma unroll
          for (int c = 0; c < kBN; ++c)
            if (key0 + c > limit) s[c] = -CUDART_INF_F;
        }
        // row max as a tree over 8 independent partial maxima (no 128-long chain)
        float mp[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mp[e] = s[e];
#pragma unroll
        for (int c = 8; c < kBN; ++c) mp[c & 7] = fmaxf(mp[c & 7], s[c]);
        const float mx = fmaxf(fmaxf(fmaxf(mp[0], mp[1]), fmaxf(mp[2], mp[3])),
                               fmaxf(fmaxf(mp[4], mp[5]), fmaxf(mp[6], mp[7])));
        const float mx_s = mx * p.scale_log2;
        const bool need = mx_s > m_ref + 8.0f;
        const float m_new = need ? mx_s : m_ref;
        const float alpha = need ? ex2_approx(m_ref - m_new) : 1.0f;
        const bool had_mass = l > 0.f;
        l *= alpha;
        m_ref = m_new;
        const float m_use = (m_ref == -CUDART_INF_F) ? 0.f : m_ref;
        float rp[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) rp[e] = 0.f;
        uint32_t pk[kBN / 2];
#pragma unroll
        for (int c = 0; c < kBN; c += 2) {
          const float p0 = ex2_approx(fmaf(s[c], p.scale_log2, -m_use));
          const float p1 = ex2_approx(fmaf(s[c + 1], p.scale_log2, -m_use));
          rp[(c >> 1) & 7] += p0 + p1;
          pk[c / 2] = pack_bf16x2(p0, p1);
        }
        l += ((rp[0] + rp[1]) + (rp[2] + rp[3])) + ((rp[4] + rp[5]) + (rp[6] + rp[7]));
        if (i > 0 && __any_sync(0xffffffffu, need && had_mass)) {
          // O holds the sum up to the previous tile: rescale it once that PV
          // landed, before this tile's P is published.
          const bool got_o = mbar_wait(&bars->o_done, (s_it - 1) & 1, abort, p.err,
                                       CSR_DEVERR_WAIT_TIMEOUT);
          if (!__all_sync(0xffffffffu, got_o)) {
            ok = false;
            break;
          }
          tc_fence_after();
          rescale_o<HD>(tmem + lane_base + C::kOCol, alpha);
        }
        tmem_st64(tmem + lane_base + sb * kBN, pk);
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&bars->p_full[sb]);
        ++s_it;
      }
      if (!ok) break;
      // ---------------------------------------------------- epilogue
      // o_final completes once per segment; o_done could be one PV behind here.
      const bool got_o = mbar_wait(&bars->o_final, seg_n & 1, abort, p.err,
                                   CSR_DEVERR_WAIT_TIMEOUT);
      if (!__all_sync(0xffffffffu, got_o)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float inv_l = l > 0.f ? 1.0f / l : 0.f;
      const float lse2 = l > 0.f ? m_ref + log2f(l) : -CUDART_INF_F;
      uint32_t o[HD];
      load_o<HD>(tmem + lane_base + C::kOCol, o);
      if (seg.complete) {
        const int hq_idx = seg.head * p.group + row % p.group;
        uint16_t *dst = p.out + (static_cast<int64_t>(t) * p.hq + hq_idx) * HD;
        if (valid) {
#pragma unroll
          for (int q8 = 0; q8 < HD / 8; ++q8) {
            uint32_t w[4];
#pragma unroll
            for (int c = 0; c < 4; ++c)
              w[c] = pack_bf16x2(__uint_as_float(o[q8 * 8 + 2 * c]) * inv_l,
                                 __uint_as_float(o[q8 * 8 + 2 * c + 1]) * inv_l);
            reinterpret_cast<uint4 *>(dst)[q8] = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
        if (valid && p.lse) p.lse[static_cast<int64_t>(hq_idx) * p.n + t] = lse2 * 0.69314718055994531f;
      } else {
        const int64_t base = static_cast<int64_t>(seg.item) * kBM + row;
        float4 *d4 = reinterpret_cast<float4 *>(p.part_o + base * HD);
#pragma unroll
        for (int c = 0; c < HD / 4; ++c)
          d4[c] = make_float4(__uint_as_float(o[4 * c]) * inv_l, __uint_as_float(o[4 * c + 1]) * inv_l,
                              __uint_as_float(o[4 * c + 2]) * inv_l, __uint_as_float(o[4 * c + 3]) * inv_l);
        p.part_lse[base] = lse2;
      }
      tc_fence_before();
      mbar_arrive(&bars->o_free);
      ++seg_n;
    }
  }

  pdl_launch_dependents();
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ============================================================ two-tile kernel
// Same work as attn_kernel, but one CTA owns two consecutive 128-row query
// tiles (A, B) of a KV head: every K/V tile staged in shared memory feeds both,
// halving the load traffic per FLOP, and two softmax warpgroups alternate with
// the tensor core.  MMA issue order per key tile i (one thread):
//   PV_A(i), S_A(i+1), PV_B(i), S_B(i+1)
// so the commit that publishes S_X(i+1) also covers PV_X(i): a softmax
// warpgroup that sees its next scores may rescale its O without another wait.
// TMEM: S_A [0,128), S_B [128,256), O_A [256,256+d), O_B [256+d,256+2d).
// 320 threads: warps 0-3 softmax A, warps 4-7 softmax B, warp 8 TMA producer,
// warp 9 MMA issuer.
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
  static constexpr int kSmem = kPtOff + kPtStage * 4 + 1024;
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kOCol = 2 * kBN;                   // O_A; O_B at kOCol + HD
};

struct PairBars {
  uint64_t q_full, q_empty;
  uint64_t k_full[4], k_empty[4], v_full[4], v_empty[4];
  uint64_t s_full[2], p_full[2], o_final[2], o_free[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

size_t attn_pair_smem_bytes(int head_dim) {
  return head_dim == 64 ? PairCfg<64>::kSmem : PairCfg<128>::kSmem;
}

// Items of the two-tile kernel: (chunk, head, pair); the pair's key range is
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
      const int64_t kv = unit_iters(p.L, p.n, T, 2 * pair + 1, p.kv_tile);
      const int64_t j0 = static_cast<int64_t>(k) * p.chunk_tiles;
      if (j0 >= kv) continue;
      s.head = head;
      s.tile = pair;  // pair index
      s.item = it;
      s.nk = static_cast<int32_t>((kv + p.chunk_tiles - 1) / p.chunk_tiles);
      s.j0 = j0;
      s.j1 = min(j0 + p.chunk_tiles, kv);
      s.complete = kv <= p.chunk_tiles;
      return true;
    }
    return false;
  }
};

constexpr int kPairThreads = 320;

template <int HD>
__global__ void __launch_bounds__(kPairThreads, 1) attn_pair_kernel(const __grid_constant__ AttnParams p) {
  using C = PairCfg<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  PairBars *bars = reinterpret_cast<PairBars *>(smem + C::kBarOff);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int T = kBM / p.group;

  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
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
    bars->abort = 0;
    fence_barrier_init();
  }
  if (warp == 8 && lane == 0) {
    tma_prefetch_desc(&p.tm_q);
    tma_prefetch_desc(&p.tm_k);
    tma_prefetch_desc(&p.tm_v);
  }
  if (warp == 9) {
    tmem_alloc(&bars->tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();   // the block's queries, keys and page table come from the previous kernel
  const uint32_t tmem = bars->tmem_base;
  volatile int *abort = &bars->abort;
  PairWalker walk{static_cast<int32_t>(blockIdx.x)};
  Seg seg;

  if (warp == 8) {
    // ------------------------------------------------------ TMA producer
    // The whole warp runs the loop (as the MMA issuer does); the elected lane's
    // predicate gates the expect-tx arrivals and the TMA issues.
    int32_t *stage = reinterpret_cast<int32_t *>(smem + C::kPtOff);
    const int ppt = kBN / p.page_size;
    const int tiles_per_block = C::kPtStage / ppt;
    const uint32_t leader = elect_lane();
    uint32_t q_round = 0, k_it = 0, v_it = 0;
    bool ok = true;
    while (ok && walk.next(p, T, seg)) {
      if (q_round > 0)
        ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_empty, (q_round - 1) & 1, abort, p.err,
                                               CSR_DEVERR_WAIT_TIMEOUT));
      if (!ok) break;
      mbar_arrive_expect_tx_if(leader, &bars->q_full, 2 * C::kQBytes);
      const int32_t qrow = seg.head * p.rows_cap + seg.tile * 2 * kBM;
#pragma unroll
      for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int b = 0; b < C::kBoxes; ++b)
          tma_load_2d_if(leader, smem + C::kQOff + h * C::kQBytes + b * (kBM * 128), &p.tm_q,
                         &bars->q_full, b * 64, qrow + h * kBM);
      ++q_round;
      for (int64_t jb = seg.j0; ok && jb < seg.j1; jb += tiles_per_block) {
        const int64_t je = min(jb + tiles_per_block, seg.j1);
        const int npages = static_cast<int>(je - jb) * ppt;
        __syncwarp();
        for (int i = lane; i < npages; i += 32) {
          const int64_t lp = jb * ppt + i;
          int32_t phys = (lp < p.n_pages_valid) ? p.page_table[lp] : p.page_table[0];
          if (phys < 0 || phys >= p.pool_pages) {
            atomicOr(p.err, CSR_DEVERR_BAD_PAGE);
            phys = 0;
          }
          stage[i] = phys;
        }
        __syncwarp();
        for (int64_t j = jb; j < je; ++j) {
          const int32_t *phys = stage + static_cast<int>(j - jb) * ppt;
          const int ks = k_it % C::kStages;
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->k_empty[ks], ((k_it / C::kStages) & 1) ^ 1,
                                                 abort, p.err, CSR_DEVERR_WAIT_TIMEOUT));
          if (!ok) break;
          mbar_arrive_expect_tx_if(leader, &bars->k_full[ks], C::kTileBytes);
          load_kv_tile_if<HD>(leader, p, &p.tm_k, smem + C::kKOff + ks * C::kTileBytes,
                              &bars->k_full[ks], seg.head, phys);
          ++k_it;
          const int vs = v_it % C::kStages;
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->v_empty[vs], ((v_it / C::kStages) & 1) ^ 1,
                                                 abort, p.err, CSR_DEVERR_WAIT_TIMEOUT));
          if (!ok) break;
          mbar_arrive_expect_tx_if(leader, &bars->v_full[vs], C::kTileBytes);
          load_kv_tile_if<HD>(leader, p, &p.tm_v, smem + C::kVOff + vs * C::kTileBytes,
                              &bars->v_full[vs], seg.head, phys);
          ++v_it;
        }
      }
    }
    if (!ok && lane == 0) {
      if (q_round > 0) drain_wait(&bars->q_full, (q_round - 1) & 1);
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
    auto wait = [&](uint64_t *bar, uint32_t parity) {
      if (ok)
        ok = __all_sync(0xffffffffu, mbar_wait(bar, parity, abort, p.err, CSR_DEVERR_WAIT_TIMEOUT));
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
    while (ok && walk.next(p, T, seg)) {
      const int tile = seg.tile * 2 + wg;
      const int64_t t = static_cast<int64_t>(tile) * T + row / p.group;
      const bool valid = tile < p.n_tiles && t < p.n;
      const int64_t limit = valid ? p.L + t : -1;
      float m_ref = -CUDART_INF_F;
      float l = 0.f;
      const int nj = static_cast<int>(seg.j1 - seg.j0);
      for (int i = 0; i < nj; ++i) {
        const int64_t j = seg.j0 + i;
        const bool got = mbar_wait(&bars->s_full[wg], s_it & 1, abort, p.err,
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
        const float mx_s = mx * p.scale_log2;
        const bool need = mx_s > m_ref + 8.0f;
        const float m_new = need ? mx_s : m_ref;
        const float alpha = need ? ex2_approx(m_ref - m_new) : 1.0f;
        const bool had_mass = l > 0.f;
        l *= alpha;
        m_ref = m_new;
        const float m_use = (m_ref == -CUDART_INF_F) ? 0.f : m_ref;
        // p = 2^(s * scale_log2 - m): the scale-and-shift and the row sum run
        // on packed fp32 pairs, the exponentials one lane at a time.
        const uint64_t scale2 = f32x2(p.scale_log2, p.scale_log2);
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
      const bool got_o = mbar_wait(&bars->o_final[wg], seg_n & 1, abort, p.err,
                                   CSR_DEVERR_WAIT_TIMEOUT);
      if (!__all_sync(0xffffffffu, got_o)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float inv_l = l > 0.f ? 1.0f / l : 0.f;
      const float lse2 = l > 0.f ? m_ref + log2f(l) : -CUDART_INF_F;
      uint32_t o[HD];
      load_o<HD>(tmem + lane_base + o_col, o);
      if (seg.complete) {
        if (valid) {
          const int hq_idx = seg.head * p.group + row % p.group;
          uint16_t *dst = p.out + (static_cast<int64_t>(t) * p.hq + hq_idx) * HD;
#pragma unroll
          for (int q8 = 0; q8 < HD / 8; ++q8) {
            uint32_t w[4];
#pragma unroll
            for (int c = 0; c < 4; ++c)
              w[c] = pack_bf16x2(__uint_as_float(o[q8 * 8 + 2 * c]) * inv_l,
                                 __uint_as_float(o[q8 * 8 + 2 * c + 1]) * inv_l);
            reinterpret_cast<uint4 *>(dst)[q8] = make_uint4(w[0], w[1], w[2], w[3]);
          }
          if (p.lse) p.lse[static_cast<int64_t>(hq_idx) * p.n + t] = lse2 * 0.69314718055994531f;
        }
      } else {
        const int64_t base = static_cast<int64_t>(seg.item) * (2 * kBM) + wg * kBM + row;
        // the partial buffer is 256-byte aligned and rows are HD floats: 32-byte stores
        float *dst = p.part_o + base * HD;
#pragma unroll
        for (int c = 0; c < HD / 8; ++c) {
          uint32_t w[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) w[e] = __float_as_uint(__uint_as_float(o[8 * c + e]) * inv_l);
          st_global_v8(dst + 8 * c, w);
        }
        p.part_lse[base] = lse2;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->o_free[wg]);
      ++seg_n;
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

// ============================================================ pipelined two-tile kernel
// Two 128-row query tiles per CTA as in attn_pair_kernel, but 64-key tiles,
// which leaves TMEM room for two score buffers per query tile:
//   S_A0 [0,64) S_A1 [64,128) S_B0 [128,192) S_B1 [192,256)  O_A [256,256+d)  O_B [..+d)
// The MMA issuer runs two key tiles ahead: while softmax works on tile i of a
// query tile, the scores of tile i+1 already sit in the other buffer, so a
// softmax warpgroup never waits for the tensor core between its tiles.  Issue
// order per key tile i:  PV_A(i), S_A(i+2), PV_B(i), S_B(i+2)  (S_X(i+2) reuses
// the buffer PV_X(i) has just read, in issue order).
template <int HD>
struct PipeCfg {
  static constexpr int kStages = (HD == 64) ? 8 : 4;
  static constexpr int kBoxes = HD / 64;
  static constexpr int kQBytes = kBM * HD * 2;                 // one query tile
  static constexpr int kTileBytes = kBN64 * HD * 2;            // one 64-key K or V tile
  static constexpr int kQOff = 0;
  static constexpr int kKOff = 2 * kQBytes;
  static constexpr int kVOff = kKOff + kStages * kTileBytes;
  static constexpr int kBarOff = kVOff + kStages * kTileBytes;
  static constexpr int kPtOff = kBarOff + 1024;
  static constexpr int kPtStage = 512;
  static constexpr int kSmem = kPtOff + kPtStage * 4 + 1024;
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kOCol = 4 * kBN64;
};

struct PipeBars {
  uint64_t q_full, q_empty;
  uint64_t k_full[8], k_empty[8], v_full[8], v_empty[8];
  uint64_t s_full[2][2], p_full[2][2];   // [query tile][score buffer]
  uint64_t o_done[2], o_final[2], o_free[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

size_t attn_pipe_smem_bytes(int head_dim) {
  return head_dim == 64 ? PipeCfg<64>::kSmem : PipeCfg<128>::kSmem;
}

template <int HD>
__global__ void __launch_bounds__(320, 1) attn_pipe_kernel(const __grid_constant__ AttnParams p) {
  using C = PipeCfg<HD>;
  constexpr int BN = kBN64;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  PipeBars *bars = reinterpret_cast<PipeBars *>(smem + C::kBarOff);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int T = kBM / p.group;

  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->q_empty, 1);
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], 1);
      mbar_init(&bars->v_full[s], 1);
      mbar_init(&bars->v_empty[s], 1);
    }
    for (int w = 0; w < 2; ++w) {
      for (int b = 0; b < 2; ++b) {
        mbar_init(&bars->s_full[w][b], 1);
        mbar_init(&bars->p_full[w][b], 128);
      }
      mbar_init(&bars->o_done[w], 1);
      mbar_init(&bars->o_final[w], 1);
      mbar_init(&bars->o_free[w], 128);
    }
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    fence_barrier_init();
  }
  if (warp == 8 && lane == 0) {
    tma_prefetch_desc(&p.tm_q);
    tma_prefetch_desc(&p.tm_k);
    tma_prefetch_desc(&p.tm_v);
  }
  if (warp == 9) {
    tmem_alloc(&bars->tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();   // the block's queries, keys and page table come from the previous kernel
  const uint32_t tmem = bars->tmem_base;
  volatile int *abort = &bars->abort;
  PairWalker walk{static_cast<int32_t>(blockIdx.x)};
  Seg seg{};

  if (warp == 8) {
    // ------------------------------------------------------ TMA producer
    // Order per item: K(0), K(1), then for each i: K(i+2), V(i) -- the MMA
    // issuer consumes keys two tiles ahead of values.
    int32_t *stage = reinterpret_cast<int32_t *>(smem + C::kPtOff);
    const int tiles_per_block = (C::kPtStage - 2) * p.page_size / BN;
    uint32_t q_round = 0, k_it = 0, v_it = 0;
    bool ok = true;
    auto load_k = [&](int64_t j, int64_t lp_base) {
      const int ks = k_it % C::kStages;
      if (!mbar_wait(&bars->k_empty[ks], ((k_it / C::kStages) & 1) ^ 1, abort, p.err,
                     CSR_DEVERR_WAIT_TIMEOUT))
        return false;
      mbar_arrive_expect_tx(&bars->k_full[ks], C::kTileBytes);
      load_kv_keys<HD>(p, &p.tm_k, smem + C::kKOff + ks * C::kTileBytes, BN, &bars->k_full[ks],
                       seg.head, stage, lp_base, j * BN);
      ++k_it;
      return true;
    };
    auto load_v = [&](int64_t j, int64_t lp_base) {
      const int vs = v_it % C::kStages;
      if (!mbar_wait(&bars->v_empty[vs], ((v_it / C::kStages) & 1) ^ 1, abort, p.err,
                     CSR_DEVERR_WAIT_TIMEOUT))
        return false;
      mbar_arrive_expect_tx(&bars->v_full[vs], C::kTileBytes);
      load_kv_keys<HD>(p, &p.tm_v, smem + C::kVOff + vs * C::kTileBytes, BN, &bars->v_full[vs],
                       seg.head, stage, lp_base, j * BN);
      ++v_it;
      return true;
    };
    while (ok && walk.next(p, T, seg)) {
      if (lane == 0) {
        if (q_round > 0 && !mbar_wait(&bars->q_empty, (q_round - 1) & 1, abort, p.err,
                                      CSR_DEVERR_WAIT_TIMEOUT)) {
          ok = false;
        } else {
          mbar_arrive_expect_tx(&bars->q_full, 2 * C::kQBytes);
          const int32_t qrow = seg.head * p.rows_cap + seg.tile * 2 * kBM;
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int b = 0; b < C::kBoxes; ++b)
              tma_load_2d(smem + C::kQOff + h * C::kQBytes + b * (kBM * 128), &p.tm_q,
                          &bars->q_full, b * 64, qrow + h * kBM);
          ++q_round;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      // Stage blocks of key tiles; V of a block's first two tiles may trail
      // into the next block, so each block stages its pages plus the two
      // tiles before it.
      for (int64_t jb = seg.j0; ok && jb < seg.j1; jb += tiles_per_block - 2) {
        const int64_t je = min(jb + tiles_per_block - 2, seg.j1);
        const int64_t sb = max(seg.j0, jb - 2);
        __syncwarp();
        const int64_t lp_base = stage_pages(p, stage, BN, sb, je, lane);
        __syncwarp();
        if (lane == 0) {
          for (int64_t j = jb; j < je && ok; ++j) {
            // K(j) is loaded in the step of V(j - 2); the first two K tiles lead
            if (j < seg.j0 + 2) {
              ok = load_k(j, lp_base);
              continue;
            }
            ok = load_k(j, lp_base) && load_v(j - 2, lp_base);
          }
          if (ok && je == seg.j1) {
            // values of the last two tiles
            for (int64_t j = max(seg.j0, seg.j1 - 2); j < seg.j1 && ok; ++j) ok = load_v(j, lp_base);
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
      }
    }
    if (!ok && lane == 0) {
      if (q_round > 0) drain_wait(&bars->q_full, (q_round - 1) & 1);
      for (uint32_t i = (k_it > C::kStages ? k_it - C::kStages : 0); i < k_it; ++i)
        drain_wait(&bars->k_full[i % C::kStages], (i / C::kStages) & 1);
      for (uint32_t i = (v_it > C::kStages ? v_it - C::kStages : 0); i < v_it; ++i)
        drain_wait(&bars->v_full[i % C::kStages], (i / C::kStages) & 1);
    }
  } else if (warp == 9) {
    if (lane == 0) {
      // ------------------------------------------------------ MMA issuer
      constexpr uint32_t idesc_s = idesc_bf16_f32(kBM, BN, false, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(kBM, HD, false, true);
      const uint32_t q_base = smem_u32(smem + C::kQOff);
      const uint32_t k_base = smem_u32(smem + C::kKOff);
      const uint32_t v_base = smem_u32(smem + C::kVOff);
      uint32_t q_round = 0, k_it = 0, v_it = 0, seg_n = 0;
      uint32_t p_cnt[2][2] = {{0, 0}, {0, 0}};
      bool ok = true;
      auto wait = [&](uint64_t *bar, uint32_t parity) {
        if (ok && !mbar_wait(bar, parity, abort, p.err, CSR_DEVERR_WAIT_TIMEOUT)) ok = false;
        return ok;
      };
      auto issue_s = [&](int x, int buf, int ks) {
        const uint32_t qx = q_base + x * C::kQBytes;
        const uint32_t kst = k_base + ks * C::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint64_t a = sdesc_sw128(qx + (kk >> 2) * (kBM * 128) + (kk & 3) * 32, 16, 1024);
          const uint64_t b = sdesc_sw128(kst + (kk >> 2) * (BN * 128) + (kk & 3) * 32, 16, 1024);
          mma_bf16_ss(tmem + (2 * x + buf) * BN, a, b, idesc_s, kk > 0 ? 1u : 0u);
        }
        mma_commit(&bars->s_full[x][buf]);
      };
      auto issue_pv = [&](int x, int buf, int vs, bool first) {
        const uint32_t vst = v_base + vs * C::kTileBytes;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk) {
          const uint64_t b = sdesc_sw128(vst + kk * (16 * 128), BN * 128, 1024);
          mma_bf16_ts(tmem + C::kOCol + x * HD, tmem + (2 * x + buf) * BN + kk * 8, b, idesc_pv,
                      (!first || kk > 0) ? 1u : 0u);
        }
      };
      while (ok && walk.next(p, T, seg)) {
        if (!wait(&bars->q_full, q_round & 1)) break;
        ++q_round;
        tc_fence_after();
        const int nj = static_cast<int>(seg.j1 - seg.j0);
        const int lead = nj < 2 ? nj : 2;
        for (int t = 0; t < lead && ok; ++t) {
          const int ks = k_it % C::kStages;
          if (!wait(&bars->k_full[ks], (k_it / C::kStages) & 1)) break;
          tc_fence_after();
          issue_s(0, t, ks);
          issue_s(1, t, ks);
          mma_commit(&bars->k_empty[ks]);
          ++k_it;
        }
        if (!ok) break;
        if (nj <= 2) mma_commit(&bars->q_empty);
        for (int i = 0; i < nj; ++i) {
          const int buf = i & 1;
          const int vs = v_it % C::kStages;
          const bool more = i + 2 < nj;
          int ks = 0;
          // ---- tile A
          if (!wait(&bars->p_full[0][buf], p_cnt[0][buf] & 1)) break;
          ++p_cnt[0][buf];
          if (!wait(&bars->v_full[vs], (v_it / C::kStages) & 1)) break;
          if (i == 0 && seg_n > 0 && !wait(&bars->o_free[0], (seg_n & 1) ^ 1)) break;
          tc_fence_after();
          issue_pv(0, buf, vs, i == 0);
          mma_commit(&bars->o_done[0]);
          if (i == nj - 1) mma_commit(&bars->o_final[0]);
          if (more) {
            ks = k_it % C::kStages;
            if (!wait(&bars->k_full[ks], (k_it / C::kStages) & 1)) break;
            tc_fence_after();
            issue_s(0, buf, ks);
          }
          // ---- tile B
          if (!wait(&bars->p_full[1][buf], p_cnt[1][buf] & 1)) break;
          ++p_cnt[1][buf];
          if (i == 0 && seg_n > 0 && !wait(&bars->o_free[1], (seg_n & 1) ^ 1)) break;
          tc_fence_after();
          issue_pv(1, buf, vs, i == 0);
          mma_commit(&bars->o_done[1]);
          if (i == nj - 1) mma_commit(&bars->o_final[1]);
          mma_commit(&bars->v_empty[vs]);
          ++v_it;
          if (more) {
            issue_s(1, buf, ks);
            mma_commit(&bars->k_empty[ks]);
            ++k_it;
            if (i + 2 == nj - 1) mma_commit(&bars->q_empty);
          }
        }
        ++seg_n;
      }
      if (!ok) {
        mma_commit(&bars->drain);
        drain_wait(&bars->drain, 0);
      }
    }
  } else {
    // ------------------------------------------------------ softmax warpgroups
    const int wg = warp >> 2;
    const int row = threadIdx.x - wg * 128;
    const uint32_t lane_base = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t o_col = C::kOCol + wg * HD;
    uint32_t s_cnt[2] = {0, 0};
    uint32_t g_tiles = 0, seg_n = 0;   // tiles (= PVs) of this warpgroup so far, items
    bool ok = true;
    while (ok && walk.next(p, T, seg)) {
      const int tile = seg.tile * 2 + wg;
      const int64_t t = static_cast<int64_t>(tile) * T + row / p.group;
      const bool valid = tile < p.n_tiles && t < p.n;
      const int64_t limit = valid ? p.L + t : -1;
      float m_ref = -CUDART_INF_F;
      float l = 0.f;
      const int nj = static_cast<int>(seg.j1 - seg.j0);
      for (int i = 0; i < nj; ++i) {
        const int buf = i & 1;
        const uint32_t s_col = (2 * wg + buf) * BN;
        const int64_t j = seg.j0 + i;
        const bool got = mbar_wait(&bars->s_full[wg][buf], s_cnt[buf] & 1, abort, p.err,
                                   CSR_DEVERR_WAIT_TIMEOUT);
        ++s_cnt[buf];
        if (!__all_sync(0xffffffffu, got)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t sr[BN];
        tmem_ld64_wait(tmem + lane_base + s_col, sr);
        float s[BN];
#pragma unroll
        for (int c = 0; c < BN; ++c) s[c] = __uint_as_float(sr[c]);
        const int64_t key0 = j * BN;
        if (key0 + BN - 1 > limit) {
#pragma unroll
          for (int c = 0; c < BN; ++c)
            if (key0 + c > limit) s[c] = -CUDART_INF_F;
        }
        float mp[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mp[e] = s[e];
#pragma unroll
        for (int c = 8; c < BN; ++c) mp[c & 7] = fmaxf(mp[c & 7], s[c]);
        const float mx = fmaxf(fmaxf(fmaxf(mp[0], mp[1]), fmaxf(mp[2], mp[3])),
                               fmaxf(fmaxf(mp[4], mp[5]), fmaxf(mp[6], mp[7])));
        const float mx_s = mx * p.scale_log2;
        const bool need = mx_s > m_ref + 8.0f;
        const float m_new = need ? mx_s : m_ref;
        const float alpha = need ? ex2_approx(m_ref - m_new) : 1.0f;
        const bool had_mass = l > 0.f;
        l *= alpha;
        m_ref = m_new;
        const float m_use = (m_ref == -CUDART_INF_F) ? 0.f : m_ref;
        float rp[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) rp[e] = 0.f;
        uint32_t pk[BN / 2];
#pragma unroll
        for (int c = 0; c < BN; c += 2) {
          const float p0 = ex2_approx(fmaf(s[c], p.scale_log2, -m_use));
          const float p1 = ex2_approx(fmaf(s[c + 1], p.scale_log2, -m_use));
          rp[(c >> 1) & 7] += p0 + p1;
          pk[c / 2] = pack_bf16x2(p0, p1);
        }
        l += ((rp[0] + rp[1]) + (rp[2] + rp[3])) + ((rp[4] + rp[5]) + (rp[6] + rp[7]));
        tmem_st32(tmem + lane_base + s_col, pk);
        if (i > 0 && __any_sync(0xffffffffu, need && had_mass)) {
          // the previous tile's PV must land before O is rescaled
          const bool got_o = mbar_wait(&bars->o_done[wg], (g_tiles - 1) & 1, abort, p.err,
                                       CSR_DEVERR_WAIT_TIMEOUT);
          if (!__all_sync(0xffffffffu, got_o)) {
            ok = false;
            break;
          }
          tc_fence_after();
          rescale_o<HD>(tmem + lane_base + o_col, alpha);
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&bars->p_full[wg][buf]);
        ++g_tiles;
      }
      if (!ok) break;
      // ---------------------------------------------------- epilogue
      const bool got_o = mbar_wait(&bars->o_final[wg], seg_n & 1, abort, p.err,
                                   CSR_DEVERR_WAIT_TIMEOUT);
      if (!__all_sync(0xffffffffu, got_o)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float inv_l = l > 0.f ? 1.0f / l : 0.f;
      const float lse2 = l > 0.f ? m_ref + log2f(l) : -CUDART_INF_F;
      uint32_t o[HD];
      load_o<HD>(tmem + lane_base + o_col, o);
      if (seg.complete) {
        if (valid) {
          const int hq_idx = seg.head * p.group + row % p.group;
          uint16_t *dst = p.out + (static_cast<int64_t>(t) * p.hq + hq_idx) * HD;
#pragma unroll
          for (int q8 = 0; q8 < HD / 8; ++q8) {
            uint32_t w[4];
#pragma unroll
            for (int c = 0; c < 4; ++c)
              w[c] = pack_bf16x2(__uint_as_float(o[q8 * 8 + 2 * c]) * inv_l,
                                 __uint_as_float(o[q8 * 8 + 2 * c + 1]) * inv_l);
            reinterpret_cast<uint4 *>(dst)[q8] = make_uint4(w[0], w[1], w[2], w[3]);
          }
          if (p.lse) p.lse[static_cast<int64_t>(hq_idx) * p.n + t] = lse2 * 0.69314718055994531f;
        }
      } else {
        const int64_t base = static_cast<int64_t>(seg.item) * (2 * kBM) + wg * kBM + row;
        float4 *d4 = reinterpret_cast<float4 *>(p.part_o + base * HD);
#pragma unroll
        for (int c = 0; c < HD / 4; ++c)
          d4[c] = make_float4(__uint_as_float(o[4 * c]) * inv_l, __uint_as_float(o[4 * c + 1]) * inv_l,
                              __uint_as_float(o[4 * c + 2]) * inv_l, __uint_as_float(o[4 * c + 3]) * inv_l);
        p.part_lse[base] = lse2;
      }
      tc_fence_before();
      mbar_arrive(&bars->o_free[wg]);
      ++seg_n;
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
// Merge the key-chunk pieces of one row: lse = log2 sum_k 2^lse_k and
// O = sum_k 2^(lse_k - lse) O_k (each O_k already normalised by its own sum).
// One warp per packed row; lanes own head_dim/32 output columns.
// 32-byte global loads (the partial buffer is 256-byte aligned and its rows
// are HD floats, so every lane's eight floats start on a 32-byte boundary).
__device__ __forceinline__ void ld_global_v8f(const float *ptr, float (&v)[8]) {
  asm volatile("ld.global.v8.f32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
               : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]),
                 "=f"(v[7])
               : "l"(ptr));
}

// K3: combine the split-KV partials of every row: lse = log2(sum_k 2^lse_k),
// out = sum_k 2^(lse_k - lse) * O_k (each O_k already normalised by its own
// row sum).  A row is read by a group of HD / 8 lanes (eight floats, one
// 32-byte load per lane per chunk); a block of 256 threads holds 256 / (HD/8)
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
  const int uph = (p.n_tiles + p.unit_tiles - 1) / p.unit_tiles;  // units per head
  const int unit = tile / p.unit_tiles;
  const int half = tile - unit * p.unit_tiles;
  const int64_t kv = unit_iters(p.L, p.n, T, unit * p.unit_tiles + p.unit_tiles - 1, p.kv_tile);
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
  const int64_t rows_per_item = static_cast<int64_t>(p.unit_tiles) * kBM;
  const int64_t row_in_item = static_cast<int64_t>(half) * kBM + r;
  // row index (item * rows_per_item + row_in_item) of chunk k's partial
  auto prow = [&](int k) {
    return (static_cast<int64_t>(k) * units + static_cast<int64_t>(head) * uph + unit) * rows_per_item +
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
    float v[kC][8], lk[kC];
#pragma unroll
    for (int u = 0; u < kC; ++u) {
      const int k = sub + u * spr;
      if (valid && k < nk) {
        lk[u] = p.part_lse[prow(k)];
        ld_global_v8f(p.part_o + prow(k) * HD + sl * 8, v[u]);
      } else {
        lk[u] = -CUDART_INF_F;
#pragma unroll
        for (int e = 0; e < 8; ++e) v[u][e] = 0.f;
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
      for (int u = 0; u < kC; ++u) {
        const float w = ex2_approx(lk[u] - lse2);
#pragma unroll
        for (int x = 0; x < 8; ++x) acc[x] = fmaf(w, v[u][x], acc[x]);
      }
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
        const float w = ex2_approx(p.part_lse[base] - lse2);
        float v[8];
        ld_global_v8f(p.part_o + base * HD + sl * 8, v);
#pragma unroll
        for (int x = 0; x < 8; ++x) acc[x] = fmaf(w, v[x], acc[x]);
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
    e = cudaFuncSetAttribute(attn_kernel<64>, attr, AttnCfg<64>::kSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(attn_pair_kernel<64>, attr, PairCfg<64>::kSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(attn_pipe_kernel<64>, attr, PipeCfg<64>::kSmem);
  } else {
    e = cudaFuncSetAttribute(attn_kernel<128>, attr, AttnCfg<128>::kSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(attn_pair_kernel<128>, attr, PairCfg<128>::kSmem);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(attn_pipe_kernel<128>, attr, PipeCfg<128>::kSmem);
  }
  return e;
}

// Launch with programmatic stream serialisation (see pdl_wait).
template <typename... Args>
cudaError_t launch_pdl(void (*kernel)(Args...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       const Args &...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

cudaError_t launch_attention(const AttnParams &p, int head_dim, cudaStream_t s) {
  if (p.unit_tiles == 2 && p.kv_tile == kBN64) {
    if (head_dim == 64)
      return launch_pdl(attn_pipe_kernel<64>, dim3(p.grid), dim3(320), PipeCfg<64>::kSmem, s, p);
    return launch_pdl(attn_pipe_kernel<128>, dim3(p.grid), dim3(320), PipeCfg<128>::kSmem, s, p);
  }
  if (p.unit_tiles == 2) {
    if (head_dim == 64)
      return launch_pdl(attn_pair_kernel<64>, dim3(p.grid), dim3(kPairThreads), PairCfg<64>::kSmem, s, p);
    return launch_pdl(attn_pair_kernel<128>, dim3(p.grid), dim3(kPairThreads), PairCfg<128>::kSmem, s, p);
  }
  if (head_dim == 64)
    return launch_pdl(attn_kernel<64>, dim3(p.grid), dim3(192), AttnCfg<64>::kSmem, s, p);
  return launch_pdl(attn_kernel<128>, dim3(p.grid), dim3(192), AttnCfg<128>::kSmem, s, p);
}

cudaError_t launch_merge(const MergeParams &p, cudaStream_t s) {
  const int slots = 256 / (p.d / 8);
  const dim3 grid(p.hkv * p.n_tiles, kBM * p.slots_per_row / slots);
  if (p.d == 64) return launch_pdl(merge_kernel<64>, grid, dim3(256), 0, s, p);
  return launch_pdl(merge_kernel<128>, grid, dim3(256), 0, s, p);
}

}  // namespace csr
