// csr_noalloc.cu -- csr_attend_block_noalloc: the block path (RoPE + paged
// append, attention, split merge) for callers that cannot allocate device
// memory.  Its scratch (packed rotated queries, split-KV partials, the device
// error word) lives in one file-scope static device array instead of a
// caller-allocated workspace.
#include <cmath>
#include <cstring>
#include <mutex>

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include "../../include/csr.h"
#include "internal.h"

namespace {

using namespace csr;

constexpr size_t kQBytes = 8ull << 20;     // packed rotated queries
constexpr size_t kPartOBytes = 24ull << 20; // split partials: fp16 rows, then (from the middle) their scales
constexpr size_t kPartLseBytes = 512ull << 10;
constexpr size_t kErrBytes = 256;
constexpr size_t kScratchBytes = kQBytes + kPartOBytes + kPartLseBytes + kErrBytes;
constexpr int kMaxDevices = 64;

// One copy per device that loads the library, kept until the process exits.
// Device code could name it directly; host code must use the address that
// cudaGetSymbolAddress returns for the current device.
static __device__ __align__(256) uint8_t g_block_scratch[kScratchBytes];

struct DeviceSetup {
  bool ready = false;
  unsigned long long ctx_id = 0;  // the context the setup was made in (a reset makes a new one)
  uint8_t *scratch = nullptr;     // device address of g_block_scratch in that context
  int num_sms = 0;
};
std::mutex g_setup_mu;
DeviceSetup g_setup[kMaxDevices];

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
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

bool encode(CUtensorMap *m, const void *base, uint64_t rows, uint64_t d, uint32_t box_rows) {
  auto fn = encoder();
  if (!fn) return false;
  cuuint64_t dims[2] = {d, rows};
  cuuint64_t strides[1] = {d * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

// Unique id of the calling thread's current context (0 if none or the driver
// lacks the query).  The runtime's primary context of a device is replaced by
// cudaDeviceReset, and with it the module holding the scratch array and the
// kernels' attributes: the setup below is redone whenever the id changes.
unsigned long long current_context_id() {
  static PFN_cuCtxGetCurrent_v4000 get_current = nullptr;
  static PFN_cuCtxGetId_v12000 get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<PFN_cuCtxGetCurrent_v4000>(p);
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<PFN_cuCtxGetId_v12000>(p);
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

// With the device current: resolve the scratch array's device address and
// raise the attention kernels' shared-memory limit, once per context of the
// device.
csr_status setup_device(int dev, DeviceSetup **out) {
  if (dev < 0 || dev >= kMaxDevices) return CSR_EINVAL;
  std::lock_guard<std::mutex> lock(g_setup_mu);
  DeviceSetup &s = g_setup[dev];
  void *sym = nullptr;
  // also makes the device's primary context current on this thread
  if (cudaGetSymbolAddress(&sym, g_block_scratch) != cudaSuccess) return CSR_ECUDA;
  const unsigned long long ctx_id = current_context_id();
  if (!s.ready || ctx_id == 0 || ctx_id != s.ctx_id || sym != s.scratch) {
    s.ready = false;
    if (attn_configure(64) != cudaSuccess || attn_configure(128) != cudaSuccess) return CSR_ECUDA;
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      return CSR_ECUDA;
    s.scratch = static_cast<uint8_t *>(sym);
    s.ctx_id = ctx_id;
    s.num_sms = sms;
    s.ready = true;
  }
  *out = &s;
  return CSR_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" csr_status csr_attend_block_noalloc(const csr_block_args *a, csr_stream_t stream) {
  if (!a) return CSR_EINVAL;
  const int32_t hq = a->num_q_heads, hkv = a->num_kv_heads, d = a->head_dim, P = a->page_size;
  if (hq <= 0 || hkv <= 0 || hq % hkv) return CSR_EINVAL;
  const int32_t g = hq / hkv;
  if ((g & (g - 1)) != 0 || g > kBM) return CSR_EINVAL;
  if (d != 64 && d != 128) return CSR_EINVAL;
  if (P != 16 && P != 32 && P != 64 && P != 128) return CSR_EINVAL;
  if (a->n < 1 || a->L < 0 || a->pool_pages < 1 || !(a->rope_base > 1.0) || a->softmax_scale < 0.f)
    return CSR_EINVAL;
  if (static_cast<int64_t>(a->pool_pages) * hkv * P >= (1ll << 31)) return CSR_EINVAL;
  for (const void *p : {a->q, a->k, a->v, static_cast<const void *>(a->out)})
    if (!p || !aligned16(p)) return CSR_EINVAL;
  if (!a->k_pool || !a->v_pool || !a->page_table || !aligned16(a->k_pool) || !aligned16(a->v_pool))
    return CSR_EINVAL;
  // The packed queries of this call must fit the static scratch.  Bound each
  // factor before multiplying: max_rows is at most 2^22 and n * g at most
  // 2^38, so nothing below overflows 64 bits whatever the arguments.
  const int64_t max_rows = static_cast<int64_t>(kQBytes) / (static_cast<int64_t>(hkv) * d * 2);
  if (static_cast<int64_t>(a->n) * g > max_rows) return CSR_EINVAL;
  const int64_t rows_cap = cdiv(static_cast<int64_t>(a->n) * g, 2 * kBM) * 2 * kBM;
  if (rows_cap > max_rows) return CSR_EINVAL;
  if (a->L > (1ll << 24) - a->n) return CSR_EINVAL;   // RoPE positions stay exact fp32 integers

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return CSR_ECUDA;
  DeviceSetup *ds = nullptr;
  csr_status st = setup_device(dev, &ds);
  if (st != CSR_OK) return st;
  uint16_t *q_pack = reinterpret_cast<uint16_t *>(ds->scratch);
  // the item cap below counts 4 bytes per value, so the fp16 rows fit the
  // first half and their scales (4 bytes per row) the second
  uint16_t *part_o = reinterpret_cast<uint16_t *>(ds->scratch + kQBytes);
  float *part_scale = reinterpret_cast<float *>(ds->scratch + kQBytes + kPartOBytes / 2);
  float *part_lse = reinterpret_cast<float *>(ds->scratch + kQBytes + kPartOBytes);
  uint32_t *err = reinterpret_cast<uint32_t *>(ds->scratch + kQBytes + kPartOBytes + kPartLseBytes);
  const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // the error word accumulates with atomicOr: start every call from zero
  if (cudaMemsetAsync(err, 0, sizeof(uint32_t), s) != cudaSuccess) return CSR_ECUDA;

  // K1: rotate, append the new keys/values through the caller's page table,
  // pack the rotated queries into the scratch
  RopeAppendParams rp{};
  rp.q = static_cast<const uint16_t *>(a->q);
  rp.k = static_cast<const uint16_t *>(a->k);
  rp.v = static_cast<const uint16_t *>(a->v);
  rp.k_pool = static_cast<uint16_t *>(a->k_pool);
  rp.v_pool = static_cast<uint16_t *>(a->v_pool);
  rp.q_pack = q_pack;
  rp.page_table = const_cast<int32_t *>(a->page_table);  // read only: n_ids == 0
  rp.err = err;
  rp.pos0 = a->L;
  rp.n = a->n;
  rp.hq = hq;
  rp.hkv = hkv;
  rp.d = d;
  rp.page_size = P;
  rp.group = g;
  rp.rows_cap = static_cast<int32_t>(rows_cap);
  rp.pool_pages = a->pool_pages;
  rp.first_lp = 0;
  rp.n_ids = 0;
  const double two_pi = 6.283185307179586476925286766559;
  for (int i = 0; i < d / 2; ++i) {
    const double w = std::pow(a->rope_base, -2.0 * i / d) / two_pi;
    rp.inv_turns[i].hi = static_cast<float>(w);
    rp.inv_turns[i].lo = static_cast<float>(w - static_cast<double>(rp.inv_turns[i].hi));
  }
  if (launch_rope_append(rp, s) != cudaSuccess) return CSR_ECUDA;

  // K2: two-tile attention over keys [0, L + n)
  AttnParams ap{};
  const uint64_t pool_rows = static_cast<uint64_t>(a->pool_pages) * hkv * P;
  if (!encode(&ap.tm_q, q_pack, static_cast<uint64_t>(hkv) * rows_cap, d, kBM) ||
      !encode(&ap.tm_k, a->k_pool, pool_rows, d, P < 64 ? P : 64) ||
      !encode(&ap.tm_v, a->v_pool, pool_rows, d, P < 64 ? P : 64))
    return CSR_ECUDA;
  ap.page_table = a->page_table;
  ap.out = static_cast<uint16_t *>(a->out);
  ap.lse = a->lse;
  ap.part_o = part_o;
  ap.part_scale = part_scale;
  ap.part_lse = part_lse;
  ap.err = err;
  ap.L = a->L;
  ap.n = a->n;
  ap.hq = hq;
  ap.hkv = hkv;
  ap.group = g;
  ap.page_size = P;
  ap.rows_cap = static_cast<int32_t>(rows_cap);
  ap.n_tiles = static_cast<int32_t>(cdiv(static_cast<int64_t>(a->n) * g, kBM));
  ap.n_pages_valid = static_cast<int32_t>(cdiv(a->L + a->n, P));
  ap.pool_pages = a->pool_pages;
  const int T = kBM / g;
  const int64_t uph = cdiv(ap.n_tiles, 2);
  const int64_t units = uph * hkv;
  const int64_t kv_max = unit_iters(a->L, a->n, T, static_cast<int32_t>(uph * 2 - 1));
  // Split the key range only as far as the static partial buffer allows:
  // one chunk per unit when there are enough units to fill the SMs, else
  // the most chunks (up to one wave) whose partials fit.
  const int64_t cap_items = static_cast<int64_t>(kPartOBytes / (2ull * kBM * d * 4));
  const int64_t lse_items = static_cast<int64_t>(kPartLseBytes / (2ull * kBM * 4));
  const int64_t max_items = cap_items < lse_items ? cap_items : lse_items;
  int64_t chunks = 1;
  if (units < ds->num_sms) {
    chunks = ds->num_sms / units;
    if (chunks * units > max_items) chunks = max_items / units;
    if (chunks < 1) chunks = 1;
    if (chunks > kv_max) chunks = kv_max;
  }
  ap.chunk_tiles = static_cast<int32_t>(cdiv(kv_max, chunks));
  const int64_t n_chunks = cdiv(kv_max, ap.chunk_tiles);
  ap.n_items = static_cast<int32_t>(n_chunks * units);
  ap.grid = static_cast<int32_t>(ap.n_items < ds->num_sms ? ap.n_items : ds->num_sms);
  const double scale = a->softmax_scale > 0.f ? static_cast<double>(a->softmax_scale)
                                              : 1.0 / std::sqrt(static_cast<double>(d));
  ap.scale_log2 = static_cast<float>(scale * 1.4426950408889634);
  if (launch_attention(ap, d, s) != cudaSuccess) return CSR_ECUDA;

  // K3: merge the split partials
  if (n_chunks > 1) {
    MergeParams mp{};
    mp.part_o = part_o;
    mp.part_scale = part_scale;
    mp.part_lse = part_lse;
    mp.out = ap.out;
    mp.lse = a->lse;
    mp.L = a->L;
    mp.n = a->n;
    mp.hq = hq;
    mp.hkv = hkv;
    mp.group = g;
    mp.n_tiles = ap.n_tiles;
    mp.chunk_tiles = ap.chunk_tiles;
    mp.d = d;
    mp.slots_per_row = merge_slots_per_row(n_chunks, mp.d);
    if (launch_merge(mp, s) != cudaSuccess) return CSR_ECUDA;
  }
  return CSR_OK;
}
