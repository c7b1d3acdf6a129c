// internal.h -- kernel parameter blocks and launch functions shared by the host
// side of libcsr (csr_api.cpp) and the kernels (kernels_*.cu).  Not part of the ABI.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace csr {

// Attention tile shape: 128 packed query rows (tokens x group heads) against
// 128 keys per step.  A unit is two consecutive query tiles of one KV head (a
// pair); TMEM holds one score buffer of 128 columns and one output
// accumulator of head_dim columns per query tile.
constexpr int kBM = 128;
constexpr int kBN = 128;
constexpr int kPairRows = 2 * kBM;
constexpr int kMaxIdsPerCall = 1024;   // new pages named by one launch
constexpr int kMaxPoolWords = 2048;    // free-bitmap words a compaction launch carries
constexpr int kMaxHalfDim = 64;        // head_dim / 2 upper bound

// RoPE frequency w_i = base^(-2i/d) / (2 pi) as two fp32 words (hi + lo), so
// that the turn count of a position is formed to about 2^-25 (rope.cuh).
struct TurnSplit {
  float hi, lo;
};

// K1: RoPE + paged append (+ GQA packing of the rotated queries).
struct RopeAppendParams {
  const uint16_t *q;       // [n][hq][d] bf16
  const uint16_t *k;       // [n][hkv][d]
  const uint16_t *v;       // [n][hkv][d]
  uint16_t *k_pool;        // [pool_pages][hkv][P][d]
  uint16_t *v_pool;
  uint16_t *q_pack;        // [hkv][rows_cap][d], row = t*G + g
  int32_t *page_table;     // device page table of the version
  uint32_t *err;
  int64_t pos0;            // absolute position of token 0
  int32_t n, hq, hkv, d, page_size, group, rows_cap, pool_pages;
  int32_t first_lp;        // logical page of pos0
  int32_t n_ids;           // > 0: ids[] give the physical pages first_lp..; 0: read page_table
  TurnSplit inv_turns[kMaxHalfDim];
  int32_t ids[kMaxIdsPerCall];
};

// K2: split-KV attention of pairs of packed query tiles over the paged cache.
struct AttnParams {
  CUtensorMap tm_q;        // q_pack as [hkv * rows_cap][d], box 64 x 128
  CUtensorMap tm_k;        // k pool as [pool_pages*hkv*P][d], box 64 x P
  CUtensorMap tm_v;
  const int32_t *page_table;
  uint16_t *out;           // [n][hq][d] bf16
  float *lse;              // [hq][n] natural log, or null
  // Split partials, one row per query row of an item (pair: 2 x kBM rows):
  // the normalised output O / l scaled by its row's largest magnitude s and
  // rounded to fp16 (|value| <= 1: 2^-12 of s at most), s itself, and the
  // log2-sum-exp.  A row of zeros has s = 0.
  uint16_t *part_o;        // [rows][d] fp16 bits
  float *part_scale;       // [rows] s
  float *part_lse;         // [rows] fp32 (log2 domain)
  uint32_t *err;
  int64_t L;               // cached tokens before this call
  int32_t n, hq, hkv, group, page_size, rows_cap, n_tiles, n_pages_valid, pool_pages;
  int32_t chunk_tiles;     // key tiles per item
  int32_t n_items;         // n_chunks * hkv * pairs per head, numbered (chunk, head, pair)
  int32_t grid;            // CTAs; CTA c runs items c, c + grid, ...
  float scale_log2;        // softmax_scale * log2(e)
};

// Schedule of a fused foreground launch (attn_pair_kernel<HD, true>): the
// pieces (unit, key tiles [j0, j1)) each CTA runs, in order.  Units are
// numbered u = pair * hkv + head.  A unit cut into several pieces is merged
// by the pieces that end last in the schedule (its last group): every other
// piece writes its normalised partial rows and log2-sum-exp to a slot and
// raises that slot's flags.  A last group of one piece waits for the flags
// and combines the partials with its own accumulator; the g > 1 pieces of a
// larger last group (pieces that run at the same time) also write partials,
// then each merges a share of the unit's 256 rows over all of them.
constexpr int kMaxStepGrid = 160;
constexpr int kMaxStepPieces = 2048;    // pieces of one launch, over all CTAs
constexpr int kMaxStepIds = 256;        // new pages one fused launch may name
constexpr uint16_t kSlotNone = 0xffff;
struct StepSchedule {
  int32_t grid;          // CTAs (<= kMaxStepGrid)
  int32_t n_units;
  int32_t n_pieces;
  int32_t n_slots;       // partial slots written (0: no unit is cut)
  uint16_t first[kMaxStepGrid + 1];    // CTA c runs pieces first[c] .. first[c + 1] - 1, in order
  uint64_t piece[kMaxStepPieces];      // unit | j0 << 16 | j1 << 40
  // merges == 0: slot is the partial slot the piece writes, or kSlotNone for a
  // whole unit (written directly).  merges > 0: the piece is in its unit's
  // last group (share = k | g << 8, member k of g); g == 1: it merges the
  // partials of slots slot .. slot + merges - 1 into its own rows; g > 1: it
  // writes slot, and the unit's merges partials are slots
  // slot - (merges - g) - k .. (the last g of them the group's), of which it
  // merges rows [k * 256 / g, (k + 1) * 256 / g)
  uint16_t slot[kMaxStepPieces];
  uint16_t merges[kMaxStepPieces];
  uint16_t share[kMaxStepPieces];
};

// Fused foreground block (one cooperative launch): RoPE + paged append of the
// new keys/values, RoPE of the queries straight into shared memory, attention,
// and the merge of cut units by their last pieces.
struct StepParams {
  AttnParams a;            // tm_q, n_items, chunk_tiles unused
  CUtensorMap tm_qraw;     // q as [n][hq][d] (3-D), box {64, G, 128/G}: one query tile per column half
  const uint16_t *q;       // [n][hq][d] bf16, before RoPE
  const uint16_t *k;       // [n][hkv][d]
  const uint16_t *v;
  uint16_t *k_pool, *v_pool;
  uint32_t *sync;          // [0]: append arrivals (monotonic)
  uint32_t *flags;         // [slot][8 softmax warps]: the launch generation once written
  uint32_t append_target;  // sync[0] once every CTA of this launch has appended its share
  uint32_t gen;            // this launch's generation (never 0; stale flags hold older ones)
  int32_t first_lp, n_ids; // logical pages first_lp.. get ids[] (written to the table by CTA 0)
  int32_t new_lp;          // logical page holding position L: key tiles reaching it wait for the append
  TurnSplit inv_turns[kMaxHalfDim];
  int32_t ids[kMaxStepIds];
  StepSchedule s;
};
static_assert(sizeof(StepParams) <= 32000, "kernel parameters of the fused launch");

// K3: merge of split partials (rebuild launches and the no-allocation block path).
struct MergeParams {
  const uint16_t *part_o;  // as AttnParams
  const float *part_scale;
  const float *part_lse;
  uint16_t *out;
  float *lse;
  int64_t L;
  int32_t n, hq, hkv, group, n_tiles, chunk_tiles, d;
  int32_t slots_per_row;   // lane groups sharing one row's chunks (a power of two)
};

// K3 merge: a row's partials are read by slots of head_dim / 8 lanes, each
// with at most kMergeChunksPerSlot partial rows in flight; rows of more
// chunks are spread over 2, 4, ... slots (up to a whole block of
// 256 / (head_dim / 8) slots, which then loops over its chunks).
constexpr int kMergeChunksPerSlot = 5;
inline int32_t merge_slots_per_row(int64_t max_chunks, int head_dim) {
  const int32_t block_slots = 256 / (head_dim / 8);
  int32_t spr = 1;
  while (spr < block_slots && spr * kMergeChunksPerSlot < max_chunks) spr *= 2;
  return spr;
}

// K4: eviction / compaction: new version's page table from the free bitmap.
struct EvictParams {
  const int32_t *old_pt;
  int32_t *new_pt;
  int32_t *ids_out;        // the fresh ids taken, in logical order
  uint16_t *k_pool;
  uint16_t *v_pool;
  uint32_t *err;
  int32_t full_prefix_pages;  // shared pages copied from old_pt
  int32_t prefix_tail;        // prefix_len % P slots copied into the first fresh page
  int32_t n_new;              // fresh pages to take
  int32_t n_words;            // bitmap words
  int32_t hkv, page_size, d, pool_pages;
  uint32_t free_words[kMaxPoolWords];  // bit b of word w: page 32w+b is free
};

// Gather of cached K/V rows of a version (inspection).
struct GatherParams {
  const uint16_t *k_pool;
  const uint16_t *v_pool;
  const int32_t *page_table;
  uint16_t *k_out;
  uint16_t *v_out;
  uint32_t *err;
  int64_t pos0;
  int32_t n, hkv, d, page_size, pool_pages;
};

// Key tiles (of kBN keys) of query tile `tile`: its keys are [0, L + last token].
__host__ __device__ inline int64_t unit_iters(int64_t L, int32_t n, int32_t tokens_per_tile,
                                              int32_t tile) {
  int64_t hi = static_cast<int64_t>(tile + 1) * tokens_per_tile;
  if (hi > n) hi = n;
  return (L + hi + kBN - 1) / kBN;
}

cudaError_t launch_rope_append(const RopeAppendParams &p, cudaStream_t s);
cudaError_t launch_attention(const AttnParams &p, int head_dim, cudaStream_t s);
// Cooperative launch of the fused foreground kernel (grid = p.s.grid CTAs).
cudaError_t launch_step(const StepParams &p, int head_dim, cudaStream_t s);
cudaError_t launch_merge(const MergeParams &p, cudaStream_t s);
cudaError_t launch_evict(const EvictParams &p, cudaStream_t s);
cudaError_t launch_gather(const GatherParams &p, cudaStream_t s);
cudaError_t attn_configure(int head_dim);  // sets the dynamic shared-memory limit

}  // namespace csr
