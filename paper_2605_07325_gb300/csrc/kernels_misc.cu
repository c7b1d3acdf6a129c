// kernels_misc.cu -- the memory-bound kernels of the path:
//   K1 rope_append: rotate the new block's queries and keys at their absolute
//      positions, store keys/values into their cache slots and the rotated
//      queries into the packed per-KV-head layout the attention kernel reads;
//   K4 evict_compact: the new version's page table after an eviction (shared
//      prefix pages + the smallest free ids from a bitmap) and the copy of a
//      partly filled prefix page;
//   gather: read cached rows of a version back in token order (inspection).
#include <cuda_bf16.h>

#include "../../include/csr.h"
#include "internal.h"
#include "ptx.cuh"
#include "rope.cuh"

namespace csr {

// Block (token t, part y): the token's 16-byte work items (rotated query
// pairs, rotated key pairs, value vectors) y, y + gridDim.y, ... in units of
// 256.  Angles theta_i = pos * base^(-2i/d) from rope_cos_sin (rope.cuh: the
// turn count in two fp32 words, reduced to [-1/2, 1/2] before the fp32
// sincospi, so positions past 10^5 keep full fp32 angle accuracy).
__global__ void __launch_bounds__(256) rope_append_kernel(const __grid_constant__ RopeAppendParams p) {
  __shared__ float cs[kMaxHalfDim], sn[kMaxHalfDim];
  const int t = blockIdx.x;
  const int64_t pos = p.pos0 + t;
  const int half = p.d / 2;
  for (int i = threadIdx.x; i < half; i += blockDim.x) rope_cos_sin(pos, p.inv_turns[i], cs[i], sn[i]);
  // The previous kernel of the stream may still read the packed queries and
  // cache pages this block overwrites.
  pdl_wait();
  // The attention kernel may launch now (its setup overlaps this kernel).
  // Triggering only after the wait means that when it starts, every earlier
  // kernel of the stream has completed: it may read the cached keys before
  // position pos0 and their page-table entries at once, and waits for this
  // grid only before the queries, the new keys and the new pages.
  pdl_launch_dependents();
  if (blockIdx.x == 0 && blockIdx.y == 0 && p.n_ids > 0) {
    for (int i = threadIdx.x; i < p.n_ids; i += blockDim.x) p.page_table[p.first_lp + i] = p.ids[i];
  }
  __syncthreads();
  const int64_t lp = pos / p.page_size;
  const int off = static_cast<int>(pos % p.page_size);
  int32_t phys = p.n_ids > 0 ? p.ids[lp - p.first_lp] : p.page_table[lp];
  if (phys < 0 || phys >= p.pool_pages) {
    if (threadIdx.x == 0) atomicOr(p.err, CSR_DEVERR_BAD_PAGE);
    return;
  }
  const int c16 = p.d / 16;  // 8-pair chunks per head
  const int c8 = p.d / 8;    // 16-byte vectors per head
  const int nq = p.hq * c16, nk = p.hkv * c16, nv = p.hkv * c8;
  for (int w = blockIdx.y * blockDim.x + threadIdx.x; w < nq + nk + nv; w += gridDim.y * blockDim.x) {
    if (w < nq + nk) {
      const bool is_q = w < nq;
      const int ww = is_q ? w : w - nq;
      const int h = ww / c16;
      const int i0 = (ww % c16) * 8;
      const uint16_t *src = is_q ? p.q + (static_cast<int64_t>(t) * p.hq + h) * p.d
                                 : p.k + (static_cast<int64_t>(t) * p.hkv + h) * p.d;
      const uint4 a = *reinterpret_cast<const uint4 *>(src + i0);
      const uint4 b = *reinterpret_cast<const uint4 *>(src + i0 + half);
      uint4 ya, yb;
      rope_rotate8(a, b, cs + i0, sn + i0, ya, yb);
      uint16_t *dst;
      if (is_q) {
        const int kvh = h / p.group, g = h % p.group;
        dst = p.q_pack + (static_cast<int64_t>(kvh) * p.rows_cap + static_cast<int64_t>(t) * p.group + g) * p.d;
      } else {
        dst = p.k_pool + ((static_cast<int64_t>(phys) * p.hkv + h) * p.page_size + off) * p.d;
      }
      *reinterpret_cast<uint4 *>(dst + i0) = ya;
      *reinterpret_cast<uint4 *>(dst + i0 + half) = yb;
    } else {
      const int ww = w - nq - nk;
      const int h = ww / c8;
      const int e0 = (ww % c8) * 8;
      const uint16_t *src = p.v + (static_cast<int64_t>(t) * p.hkv + h) * p.d + e0;
      uint16_t *dst = p.v_pool + ((static_cast<int64_t>(phys) * p.hkv + h) * p.page_size + off) * p.d + e0;
      *reinterpret_cast<uint4 *>(dst) = *reinterpret_cast<const uint4 *>(src);
    }
  }
}

cudaError_t launch_rope_append(const RopeAppendParams &p, cudaStream_t s) {
  // Short blocks split each token over several CTAs (one work item per
  // thread: latency-bound otherwise); long blocks already fill the GPU with
  // one CTA per token and would only recompute the angle table.
  const int items = (p.hq + p.hkv) * (p.d / 16) + p.hkv * (p.d / 8);
  const dim3 grid(p.n, p.n < 128 ? (items + 255) / 256 : 1);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, rope_append_kernel, p);
}

// K4: one block.  Copies the shared prefix entries, takes the n_new smallest
// free ids of the bitmap snapshot in ascending order (block-wide exclusive
// scan of per-thread free counts), and copies the prefix slots of a partly
// filled last prefix page into the first fresh page.
__global__ void __launch_bounds__(1024) evict_compact_kernel(const __grid_constant__ EvictParams p) {
  __shared__ int32_t warp_tot[32];
  __shared__ int32_t tail_page;
  const int tid = threadIdx.x;
  for (int i = tid; i < p.full_prefix_pages; i += blockDim.x) p.new_pt[i] = p.old_pt[i];
  // each thread owns a contiguous run of bitmap words
  const int per = (p.n_words + blockDim.x - 1) / blockDim.x;
  const int w0 = min(tid * per, p.n_words);
  const int w1 = min(w0 + per, p.n_words);
  int mine = 0;
  for (int w = w0; w < w1; ++w) mine += __popc(p.free_words[w]);
  // exclusive scan over the block
  const int lane = tid & 31, wid = tid >> 5;
  int incl = mine;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += y;
  }
  if (lane == 31) warp_tot[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    int v = lane < (blockDim.x >> 5) ? warp_tot[lane] : 0;
    int vi = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, vi, off);
      if (lane >= off) vi += y;
    }
    warp_tot[lane] = vi - v;  // exclusive prefix of each warp
  }
  __syncthreads();
  int rank = warp_tot[wid] + incl - mine;
  if (tid == blockDim.x - 1 && rank + mine < p.n_new) atomicOr(p.err, CSR_DEVERR_ALLOC);
  for (int w = w0; w < w1 && rank < p.n_new; ++w) {
    uint32_t bits = p.free_words[w];
    while (bits && rank < p.n_new) {
      const int b = __ffs(bits) - 1;
      bits &= bits - 1;
      const int32_t id = w * 32 + b;
      p.new_pt[p.full_prefix_pages + rank] = id;
      p.ids_out[rank] = id;
      if (rank == 0) tail_page = id;
      ++rank;
    }
  }
  __syncthreads();
  if (p.prefix_tail > 0 && p.n_new > 0) {
    const int32_t src_page = p.old_pt[p.full_prefix_pages];
    const int32_t dst_page = tail_page;
    if (src_page < 0 || src_page >= p.pool_pages || dst_page < 0 || dst_page >= p.pool_pages) {
      if (tid == 0) atomicOr(p.err, CSR_DEVERR_BAD_PAGE);
      return;
    }
    const int vec_per_row = p.d / 8;
    const int rows = p.hkv * p.prefix_tail;
    for (int e = tid; e < 2 * rows * vec_per_row; e += blockDim.x) {
      const int which = e / (rows * vec_per_row);
      const int r = (e / vec_per_row) % rows;
      const int c = e % vec_per_row;
      const int h = r / p.prefix_tail, slot = r % p.prefix_tail;
      const uint16_t *base = which == 0 ? p.k_pool : p.v_pool;
      uint16_t *obase = which == 0 ? p.k_pool : p.v_pool;
      const int64_t so = ((static_cast<int64_t>(src_page) * p.hkv + h) * p.page_size + slot) * p.d + c * 8;
      const int64_t dof = ((static_cast<int64_t>(dst_page) * p.hkv + h) * p.page_size + slot) * p.d + c * 8;
      *reinterpret_cast<uint4 *>(obase + dof) = *reinterpret_cast<const uint4 *>(base + so);
    }
  }
}

cudaError_t launch_evict(const EvictParams &p, cudaStream_t s) {
  evict_compact_kernel<<<1, 1024, 0, s>>>(p);
  return cudaGetLastError();
}

__global__ void __launch_bounds__(256) gather_kernel(const __grid_constant__ GatherParams p) {
  const int t = blockIdx.x;
  const int64_t pos = p.pos0 + t;
  const int32_t phys = p.page_table[pos / p.page_size];
  const int off = static_cast<int>(pos % p.page_size);
  if (phys < 0 || phys >= p.pool_pages) {
    if (threadIdx.x == 0) atomicOr(p.err, CSR_DEVERR_BAD_PAGE);
    return;
  }
  const int vec = p.d / 8;
  for (int e = threadIdx.x; e < 2 * p.hkv * vec; e += blockDim.x) {
    const int which = e / (p.hkv * vec);
    const int h = (e / vec) % p.hkv;
    const int c = e % vec;
    const int64_t so = ((static_cast<int64_t>(phys) * p.hkv + h) * p.page_size + off) * p.d + c * 8;
    const int64_t dof = (static_cast<int64_t>(t) * p.hkv + h) * p.d + c * 8;
    if (which == 0)
      *reinterpret_cast<uint4 *>(p.k_out + dof) = *reinterpret_cast<const uint4 *>(p.k_pool + so);
    else
      *reinterpret_cast<uint4 *>(p.v_out + dof) = *reinterpret_cast<const uint4 *>(p.v_pool + so);
  }
}

cudaError_t launch_gather(const GatherParams &p, cudaStream_t s) {
  gather_kernel<<<p.n, 256, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace csr
