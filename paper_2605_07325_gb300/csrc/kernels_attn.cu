// kernels_attn.cu -- causal attention of a block of new tokens over the paged
// cache (Eq. causal_attention_1..3: a_n = softmax(q_n K_{1:n}^T / sqrt(d_k)),
// o_n = a_n V_{1:n}), on the 5th-generation tensor cores of sm_103a.
//
// Work decomposition.  The rotated queries of one KV head are packed as rows
// t*G + g (token t, group member g), so one 128-row tile holds 128/G tokens of
// all G query heads that read the same keys.  A unit is one (kv head, query
// tile); its key range is [0, L + last token of the tile], walked in tiles of
// 128 keys.  The (unit, key tile) iteration space is cut into `grid` equal
// contiguous ranges, one per CTA (stream-K): a CTA that holds a whole unit
// writes its output directly, the pieces of a unit split between CTAs are
// written as normalised partials with their log-sum-exp and merged by K3.
//
// CTA roles (192 threads):
//   warp 4 lane 0  TMA producer: the Q tile, then K and V tiles page by page
//                  (page table lookup per 64/16-token page), into 128-byte
//                  swizzled shared memory rings;
//   warp 5 lane 0  MMA issuer: S = Q K^T into one of two TMEM score buffers
//                  (tcgen05.mma, both operands in shared memory), then
//                  O += P V with P read from TMEM and V from shared memory;
//   warps 0-3      softmax: one thread per query row (its TMEM lane); masks
//                  keys past the row's position, keeps a running max with a
//                  lazy rescale of O (only when the max grows by more than
//                  2^8), writes P as bf16 over its own score columns, and
//                  finally normalises O and stores it.
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
  static constexpr int kSmem = kBarOff + 1024 + 1024;    // barriers + alignment slack
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
  int32_t start_head, start_tile;
  int64_t start_j;
};

size_t attn_smem_bytes(int head_dim) {
  return head_dim == 64 ? AttnCfg<64>::kSmem : AttnCfg<128>::kSmem;
}

// One contiguous run of key tiles of one unit inside a CTA's range.
struct Seg {
  int32_t head, tile;
  int64_t j0, j1;
  bool complete, first;
};

struct SegWalker {
  int32_t head, tile;
  int64_t j, g, g0, g1;
  __device__ bool next(const AttnParams &p, int T, Seg &s) {
    if (g >= g1) return false;
    const int64_t it = unit_iters(p.L, p.n, T, tile);
    const int64_t take = min(it - j, g1 - g);
    s.head = head;
    s.tile = tile;
    s.j0 = j;
    s.j1 = j + take;
    s.complete = (j == 0 && take == it);
    s.first = (g == g0);
    g += take;
    j += take;
    if (j == it) {
      j = 0;
      if (++tile == p.n_tiles) {
        tile = 0;
        ++head;
      }
    }
    return true;
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

template <int HD>
__device__ __forceinline__ void load_kv_tile(const AttnParams &p, const CUtensorMap *map,
                                             uint8_t *dst, uint64_t *bar, int head, int64_t j) {
  const int P = p.page_size;
  const int ppt = kBN / P;
  const int64_t lp0 = j * kBN / P;
  for (int pp = 0; pp < ppt; ++pp) {
    const int64_t lp = lp0 + pp;
    int32_t phys = (lp < p.n_pages_valid) ? p.page_table[lp] : p.page_table[0];
    if (phys < 0 || phys >= p.pool_pages) {
      atomicOr(p.err, CSR_DEVERR_BAD_PAGE);
      phys = 0;
    }
    const int32_t row = (phys * p.hkv + head) * P;
#pragma unroll
    for (int b = 0; b < AttnCfg<HD>::kBoxes; ++b)
      tma_load_2d(dst + b * (kBN * 128) + pp * P * 128, map, bar, b * 64, row);
  }
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
  const int64_t g0 = static_cast<int64_t>(blockIdx.x) * p.total_iters / p.grid;
  const int64_t g1 = static_cast<int64_t>(blockIdx.x + 1) * p.total_iters / p.grid;

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
  if (warp == 4) {
    // Locate the CTA's first iteration: head, query tile and key tile.
    const int64_t head = g0 / p.iters_per_head;
    const int64_t rem = g0 - head * p.iters_per_head;
    const int per = (p.n_tiles + 31) / 32;
    const int t_begin = min(lane * per, p.n_tiles);
    const int t_end = min(t_begin + per, p.n_tiles);
    int64_t mine = 0;
    for (int t = t_begin; t < t_end; ++t) mine += unit_iters(p.L, p.n, T, t);
    int64_t incl = mine;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int64_t y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    const int64_t excl = incl - mine;
    const unsigned owner_mask = __ballot_sync(0xffffffffu, excl <= rem && rem < incl);
    const int owner = __ffs(owner_mask) - 1;
    if (lane == owner) {
      int64_t c = excl;
      for (int t = t_begin; t < t_end; ++t) {
        const int64_t it = unit_iters(p.L, p.n, T, t);
        if (rem < c + it) {
          bars->start_head = static_cast<int32_t>(head);
          bars->start_tile = t;
          bars->start_j = rem - c;
          break;
        }
        c += it;
      }
    }
    if (lane == 0) {
      tma_prefetch_desc(&p.tm_q);
      tma_prefetch_desc(&p.tm_k);
      tma_prefetch_desc(&p.tm_v);
    }
  }
  if (warp == 5) {
    tmem_alloc(&bars->tmem_base, C::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  volatile int *abort = &bars->abort;
  SegWalker walk{bars->start_head, bars->start_tile, bars->start_j, g0, g0, g1};
  Seg seg;

  if (warp == 4) {
    if (lane == 0) {
      // ------------------------------------------------------ TMA producer
      uint32_t q_round = 0, k_it = 0, v_it = 0;
      bool ok = true;
      while (ok && walk.next(p, T, seg)) {
        if (q_round > 0 && !mbar_wait(&bars->q_empty, (q_round - 1) & 1, abort, p.err,
                                      CSR_DEVERR_WAIT_TIMEOUT)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&bars->q_full, C::kQBytes);
        const int32_t qrow = seg.head * p.rows_cap + seg.tile * kBM;
#pragma unroll
        for (int b = 0; b < C::kBoxes; ++b)
          tma_load_2d(smem + C::kQOff + b * (kBM * 128), &p.tm_q, &bars->q_full, b * 64, qrow);
        ++q_round;
        for (int64_t j = seg.j0; j < seg.j1; ++j) {
          const int ks = k_it % C::kStages;
          if (!mbar_wait(&bars->k_empty[ks], ((k_it / C::kStages) & 1) ^ 1, abort, p.err,
                         CSR_DEVERR_WAIT_TIMEOUT)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&bars->k_full[ks], C::kTileBytes);
          load_kv_tile<HD>(p, &p.tm_k, smem + C::kKOff + ks * C::kTileBytes, &bars->k_full[ks],
                           seg.head, j);
          ++k_it;
          const int vs = v_it % C::kStages;
          if (!mbar_wait(&bars->v_empty[vs], ((v_it / C::kStages) & 1) ^ 1, abort, p.err,
                         CSR_DEVERR_WAIT_TIMEOUT)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&bars->v_full[vs], C::kTileBytes);
          load_kv_tile<HD>(p, &p.tm_v, smem + C::kVOff + vs * C::kTileBytes, &bars->v_full[vs],
                           seg.head, j);
          ++v_it;
        }
      }
      if (!ok) {
        // Let the copies already issued land before the CTA's memory goes away.
        if (q_round > 0) drain_wait(&bars->q_full, (q_round - 1) & 1);
        for (uint32_t i = (k_it > C::kStages ? k_it - C::kStages : 0); i < k_it; ++i)
          drain_wait(&bars->k_full[i % C::kStages], (i / C::kStages) & 1);
        for (uint32_t i = (v_it > C::kStages ? v_it - C::kStages : 0); i < v_it; ++i)
          drain_wait(&bars->v_full[i % C::kStages], (i / C::kStages) & 1);
      }
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
#pragma unroll
        for (int q4 = 0; q4 < kBN / 32; ++q4)
          tmem_ld32_wait(tmem + lane_base + sb * kBN + q4 * 32,
                         *reinterpret_cast<uint32_t(*)[32]>(&sr[q4 * 32]));
        float s[kBN];
#pragma unroll
        for (int c = 0; c < kBN; ++c) s[c] = __uint_as_float(sr[c]);
        const int64_t key0 = j * kBN;
        if (key0 + kBN - 1 > limit) {
#pragma unroll
          for (int c = 0; c < kBN; ++c)
            if (key0 + c > limit) s[c] = -CUDART_INF_F;
        }
        float mx = -CUDART_INF_F;
#pragma unroll
        for (int c = 0; c < kBN; ++c) mx = fmaxf(mx, s[c]);
        const float mx_s = mx * p.scale_log2;
        const bool need = mx_s > m_ref + 8.0f;
        const float m_new = need ? mx_s : m_ref;
        const float alpha = need ? ex2_approx(m_ref - m_new) : 1.0f;
        if (i > 0 && __any_sync(0xffffffffu, need && l > 0.f)) {
          // O holds the sum up to the previous tile: rescale it once that PV landed.
          const bool got_o = mbar_wait(&bars->o_done, (s_it - 1) & 1, abort, p.err,
                                       CSR_DEVERR_WAIT_TIMEOUT);
          if (!__all_sync(0xffffffffu, got_o)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int q4 = 0; q4 < HD / 32; ++q4) {
            uint32_t o[32];
            tmem_ld32_wait(tmem + lane_base + C::kOCol + q4 * 32, o);
#pragma unroll
            for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * alpha);
            tmem_st32(tmem + lane_base + C::kOCol + q4 * 32, o);
          }
          tmem_st_wait();
        }
        l *= alpha;
        m_ref = m_new;
        const float m_use = (m_ref == -CUDART_INF_F) ? 0.f : m_ref;
        float rs = 0.f;
        uint32_t pk[kBN / 2];
#pragma unroll
        for (int c = 0; c < kBN; c += 2) {
          const float p0 = ex2_approx(fmaf(s[c], p.scale_log2, -m_use));
          const float p1 = ex2_approx(fmaf(s[c + 1], p.scale_log2, -m_use));
          rs += p0 + p1;
          pk[c / 2] = pack_bf16x2(p0, p1);
        }
        l += rs;
        tmem_st32(tmem + lane_base + sb * kBN, *reinterpret_cast<uint32_t(*)[32]>(&pk[0]));
        tmem_st32(tmem + lane_base + sb * kBN + 32, *reinterpret_cast<uint32_t(*)[32]>(&pk[32]));
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
      if (seg.complete) {
        const int hq_idx = seg.head * p.group + row % p.group;
        uint16_t *dst = p.out + (static_cast<int64_t>(t) * p.hq + hq_idx) * HD;
#pragma unroll
        for (int q4 = 0; q4 < HD / 32; ++q4) {
          uint32_t o[32];
          tmem_ld32_wait(tmem + lane_base + C::kOCol + q4 * 32, o);
          if (valid) {
            uint32_t w[16];
#pragma unroll
            for (int c = 0; c < 16; ++c)
              w[c] = pack_bf16x2(__uint_as_float(o[2 * c]) * inv_l,
                                 __uint_as_float(o[2 * c + 1]) * inv_l);
            uint4 *d4 = reinterpret_cast<uint4 *>(dst + q4 * 32);
#pragma unroll
            for (int c = 0; c < 4; ++c) d4[c] = make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
          }
        }
        if (valid && p.lse) p.lse[static_cast<int64_t>(hq_idx) * p.n + t] = lse2 * 0.69314718055994531f;
      } else {
        const int slot = seg.first ? 0 : 1;
        const int64_t base = (static_cast<int64_t>(blockIdx.x) * 2 + slot) * kBM + row;
        float *dst = p.part_o + base * HD;
#pragma unroll
        for (int q4 = 0; q4 < HD / 32; ++q4) {
          uint32_t o[32];
          tmem_ld32_wait(tmem + lane_base + C::kOCol + q4 * 32, o);
          float4 *d4 = reinterpret_cast<float4 *>(dst + q4 * 32);
#pragma unroll
          for (int c = 0; c < 8; ++c)
            d4[c] = make_float4(__uint_as_float(o[4 * c]) * inv_l, __uint_as_float(o[4 * c + 1]) * inv_l,
                                __uint_as_float(o[4 * c + 2]) * inv_l, __uint_as_float(o[4 * c + 3]) * inv_l);
        }
        p.part_lse[base] = lse2;
      }
      tc_fence_before();
      mbar_arrive(&bars->o_free);
      ++seg_n;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ------------------------------------------------------------------ K3 merge
__device__ __forceinline__ int64_t cta_start(int64_t c, int64_t total, int64_t grid) {
  return c * total / grid;
}
__device__ __forceinline__ int64_t cta_of(int64_t g, int64_t total, int64_t grid) {
  int64_t c = ((g + 1) * grid - 1) / total;
  return c < grid - 1 ? c : grid - 1;
}

// Merge the split pieces of one unit: lse = log2 sum_s 2^lse_s,
// O = sum_s 2^(lse_s - lse) O_s (each O_s already normalised by its own sum).
template <int HD>
__global__ void __launch_bounds__(256) merge_kernel(const __grid_constant__ MergeParams p) {
  const int u = blockIdx.x;
  const int head = u / p.n_tiles;
  const int tile = u % p.n_tiles;
  const int T = kBM / p.group;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ int64_t s_cum;
  if (warp == 0) {
    const int per = (tile + 31) / 32;
    const int t_begin = min(lane * per, tile);
    const int t_end = min(t_begin + per, tile);
    int64_t mine = 0;
    for (int t = t_begin; t < t_end; ++t) mine += unit_iters(p.L, p.n, T, t);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mine += __shfl_xor_sync(0xffffffffu, mine, off);
    if (lane == 0) s_cum = mine;
  }
  __syncthreads();
  const int64_t us = static_cast<int64_t>(head) * p.iters_per_head + s_cum;
  const int64_t ue = us + unit_iters(p.L, p.n, T, tile);
  const int64_t c_first = cta_of(us, p.total_iters, p.grid);
  const int64_t c_last = cta_of(ue - 1, p.total_iters, p.grid);
  if (c_first == c_last) return;  // written whole by one CTA
  constexpr int kPer = HD / 32;   // floats per lane
  for (int r = warp; r < kBM; r += 8) {
    const int64_t t = static_cast<int64_t>(tile) * T + r / p.group;
    if (t >= p.n) continue;
    float mx = -CUDART_INF_F;
    for (int64_t c = c_first; c <= c_last; ++c) {
      const int slot = cta_start(c, p.total_iters, p.grid) >= us ? 0 : 1;
      mx = fmaxf(mx, p.part_lse[(c * 2 + slot) * kBM + r]);
    }
    float acc[kPer];
#pragma unroll
    for (int e = 0; e < kPer; ++e) acc[e] = 0.f;
    float lse2 = -CUDART_INF_F;
    if (mx != -CUDART_INF_F) {
      float sum = 0.f;
      for (int64_t c = c_first; c <= c_last; ++c) {
        const int slot = cta_start(c, p.total_iters, p.grid) >= us ? 0 : 1;
        sum += ex2_approx(p.part_lse[(c * 2 + slot) * kBM + r] - mx);
      }
      lse2 = mx + log2f(sum);
      for (int64_t c = c_first; c <= c_last; ++c) {
        const int slot = cta_start(c, p.total_iters, p.grid) >= us ? 0 : 1;
        const int64_t base = (c * 2 + slot) * kBM + r;
        const float w = ex2_approx(p.part_lse[base] - lse2);
        const float *src = p.part_o + base * HD + lane * kPer;
#pragma unroll
        for (int e = 0; e < kPer; ++e) acc[e] = fmaf(w, src[e], acc[e]);
      }
    }
    const int hq_idx = head * p.group + r % p.group;
    uint16_t *dst = p.out + (t * p.hq + hq_idx) * HD + lane * kPer;
#pragma unroll
    for (int e = 0; e < kPer; e += 2) {
      *reinterpret_cast<uint32_t *>(dst + e) = pack_bf16x2(acc[e], acc[e + 1]);
    }
    if (lane == 0 && p.lse) p.lse[static_cast<int64_t>(hq_idx) * p.n + t] = lse2 * 0.69314718055994531f;
  }
}

cudaError_t attn_configure(int head_dim) {
  if (head_dim == 64)
    return cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                AttnCfg<64>::kSmem);
  return cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              AttnCfg<128>::kSmem);
}

cudaError_t launch_attention(const AttnParams &p, int head_dim, cudaStream_t s) {
  if (head_dim == 64)
    attn_kernel<64><<<p.grid, 192, AttnCfg<64>::kSmem, s>>>(p);
  else
    attn_kernel<128><<<p.grid, 192, AttnCfg<128>::kSmem, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_merge(const MergeParams &p, cudaStream_t s) {
  const int units = p.hkv * p.n_tiles;
  if (p.d == 64)
    merge_kernel<64><<<units, 256, 0, s>>>(p);
  else
    merge_kernel<128><<<units, 256, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace csr
