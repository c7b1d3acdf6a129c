// internal.h -- kernel parameter blocks and launch functions shared by the host
// side of libcsr (csr_api.cpp) and the kernels (kernels_*.cu).  Not part of the ABI.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace csr {

// Attention tile shape: 128 packed query rows (tokens x group heads) against
// 128 keys per step.  TMEM: two score buffers of 128 columns and one output
// accumulator of head_dim columns.
constexpr int kBM = 128;
constexpr int kBN = 128;
constexpr int kMaxIdsPerCall = 1024;   // new pages named by one rope/append launch
constexpr int kMaxPoolWords = 2048;    // free-bitmap words a compaction launch carries
constexpr int kMaxHalfDim = 64;        // head_dim / 2 upper bound

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
  double inv_turns[kMaxHalfDim];  // base^(-2i/d) / (2 pi), i < d/2
  int32_t ids[kMaxIdsPerCall];
};

// K2: split-KV attention of the packed query tiles over the paged cache.
struct AttnParams {
  CUtensorMap tm_q;        // q_pack as [hkv * rows_cap][d], box 64 x 128
  CUtensorMap tm_k;        // k pool as [pool_pages*hkv*P][d], box 64 x P
  CUtensorMap tm_v;
  const int32_t *page_table;
  uint16_t *out;           // [n][hq][d] bf16
  float *lse;              // [hq][n] natural log, or null
  float *part_o;           // [n_items][kBM][d] fp32 (normalised partial outputs)
  float *part_lse;         // [n_items][kBM] fp32 (log2 domain)
  uint32_t *err;
  int64_t L;               // cached tokens before this call
  int32_t n, hq, hkv, group, page_size, rows_cap, n_tiles, n_pages_valid, pool_pages;
  int32_t chunk_tiles;     // key tiles per item
  int32_t unit_tiles;      // query tiles per item: 1 (attn_kernel) or 2 (pair / pipe kernels)
  int32_t kv_tile;         // keys per key tile: 128, or 64 for attn_pipe_kernel
  int32_t n_items;         // n_chunks * hkv * units per head, numbered (chunk, head, unit)
  int32_t grid;            // CTAs; CTA c runs items c, c + grid, ...
  float scale_log2;        // softmax_scale * log2(e)
};

// K3: merge of split partials.
struct MergeParams {
  const float *part_o;
  const float *part_lse;
  uint16_t *out;
  float *lse;
  int64_t L;
  int32_t n, hq, hkv, group, n_tiles, chunk_tiles, unit_tiles, kv_tile, d;
  int32_t slots_per_row;   // lane groups sharing one row's chunks (a power of two)
};

// K3 merge: a row's partials are read by slots of head_dim / 8 lanes, each
// with at most kMergeChunksPerSlot partial rows in flight; rows of more
// chunks are spread over 2, 4, ... slots (up to a whole block of
// 256 / (head_dim / 8) slots, which then loops over its chunks).
constexpr int kMergeChunksPerSlot = 4;
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

// Shared-memory bytes of the attention kernels for a head dim.
size_t attn_smem_bytes(int head_dim);
size_t attn_pair_smem_bytes(int head_dim);
size_t attn_pipe_smem_bytes(int head_dim);

// Key tiles (of `bn` keys) of query tile `tile`: its keys are [0, L + last token].
__host__ __device__ inline int64_t unit_iters(int64_t L, int32_t n, int32_t tokens_per_tile,
                                              int32_t tile, int32_t bn = kBN) {
  int64_t hi = static_cast<int64_t>(tile + 1) * tokens_per_tile;
  if (hi > n) hi = n;
  return (L + hi + bn - 1) / bn;
}

// Key tile of the pipelined kernel (attn_pipe_kernel): 64 keys, so two score
// buffers per query tile fit TMEM next to the two output accumulators.
constexpr int kBN64 = 64;

cudaError_t launch_rope_append(const RopeAppendParams &p, cudaStream_t s);
cudaError_t launch_attention(const AttnParams &p, int head_dim, cudaStream_t s);
cudaError_t launch_merge(const MergeParams &p, cudaStream_t s);
cudaError_t launch_evict(const EvictParams &p, cudaStream_t s);
cudaError_t launch_gather(const GatherParams &p, cudaStream_t s);
cudaError_t attn_configure(int head_dim);  // sets the dynamic shared-memory limit

}  // namespace csr
