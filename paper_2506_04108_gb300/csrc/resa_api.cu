// C ABI of libresa (declared in include/resa.h): host-side validation,
// workspace layout, tensor-map encoding and kernel dispatch. Every argument is
// checked before the first CUDA call, so invalid calls launch nothing and need
// no GPU.
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "resa.h"
#include "resa_launch.h"

namespace resa {
namespace {

constexpr int kMaxDevices = 64;
constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

std::atomic<int> g_sm_count[kMaxDevices];
static_assert(RESA_DEFAULT_DECODE_WAIT_POLLS == (1u << 22), "the decode's default wait bound is the kernels' own");
std::atomic<uint32_t> g_decode_wait_polls{RESA_DEFAULT_DECODE_WAIT_POLLS};

resa_status_t sm_count(int* out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return RESA_ERR_CUDA;
  if (dev < kMaxDevices) {
    const int cached = g_sm_count[dev].load(std::memory_order_relaxed);
    if (cached > 0) {
      *out = cached;
      return RESA_OK;
    }
  }
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return RESA_ERR_CUDA;
  if (dev < kMaxDevices) g_sm_count[dev].store(n, std::memory_order_relaxed);
  *out = n;
  return RESA_OK;
}

// cuTensorMapEncodeTiled through the runtime's driver entry point (no -lcuda).
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static std::atomic<EncodeTiledFn> fn{nullptr};
  EncodeTiledFn f = fn.load(std::memory_order_acquire);
  if (f != nullptr) return f;
  void* p = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || p == nullptr)
    return nullptr;
  f = reinterpret_cast<EncodeTiledFn>(p);
  fn.store(f, std::memory_order_release);
  return f;
}

// The pool viewed as a 2-D bf16 tensor [num_pages * Hkv * 16 rows][128 cols];
// a box is one 64-column half of one page of one head (16 rows x 128 bytes),
// written to shared memory with the 128-byte swizzle.
resa_status_t pool_tensor_map(const resa_cache_t* c, void* base, CUtensorMap* tm) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return RESA_ERR_CUDA;
  const cuuint64_t rows = static_cast<cuuint64_t>(c->num_pages) * c->num_kv_heads * c->block_size;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(c->head_dim), rows};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(c->head_dim) * 2};
  const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(c->block_size)};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? RESA_OK : RESA_ERR_CUDA;
}

// k_new / v_new of a rectification viewed as a 4-D bf16 tensor
// [B][f][Hkv][128] (innermost first: dim, head, token, sequence); a box is 64
// dims x 1 head x 64 tokens (one swizzled half of a 64-key tile), tokens past
// f read as zero.
resa_status_t new_kv_tensor_map(const resa_cache_t* c, const void* base, int f, CUtensorMap* tm) {
  EncodeTiledFn enc = encode_fn();
  if (enc == nullptr) return RESA_ERR_CUDA;
  const cuuint64_t row = static_cast<cuuint64_t>(c->head_dim) * 2;
  const cuuint64_t dims[4] = {static_cast<cuuint64_t>(c->head_dim), static_cast<cuuint64_t>(c->num_kv_heads),
                              static_cast<cuuint64_t>(f), static_cast<cuuint64_t>(c->batch)};
  const cuuint64_t strides[3] = {row, row * c->num_kv_heads, row * c->num_kv_heads * f};
  const cuuint32_t box[4] = {64, 1, 64, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  const CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
                         CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? RESA_OK : RESA_ERR_CUDA;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

resa_status_t check_cache(const resa_cache_t* c) {
  if (c == nullptr) return RESA_ERR_INVALID_ARG;
  if (c->batch <= 0 || c->num_q_heads <= 0 || c->num_kv_heads <= 0 || c->num_pages <= 0 ||
      c->max_blocks_per_seq <= 0)
    return RESA_ERR_INVALID_ARG;
  if (c->head_dim != kHeadDimHost || c->block_size != kBlockHost) return RESA_ERR_UNSUPPORTED;
  if (c->num_q_heads % c->num_kv_heads != 0) return RESA_ERR_INVALID_ARG;
  const int g = c->num_q_heads / c->num_kv_heads;
  if (g > 8) return RESA_ERR_UNSUPPORTED;
  // row coordinates of the pool and 32-bit index arithmetic must not overflow
  if (static_cast<int64_t>(c->num_pages) * c->num_kv_heads * c->block_size > INT32_MAX) return RESA_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(c->max_blocks_per_seq) * c->block_size > INT32_MAX / 2) return RESA_ERR_UNSUPPORTED;
  if (c->max_blocks_per_seq > select_max_blocks()) return RESA_ERR_UNSUPPORTED;
  if (c->batch > 1024) return RESA_ERR_UNSUPPORTED;
  if (c->k_pool == nullptr || c->v_pool == nullptr || c->page_table == nullptr || c->seq_lens == nullptr ||
      c->summaries == nullptr || c->device_status == nullptr)
    return RESA_ERR_INVALID_ARG;
  if (!aligned16(c->k_pool) || !aligned16(c->v_pool) || !aligned16(c->summaries)) return RESA_ERR_INVALID_ARG;
  return RESA_OK;
}

resa_status_t check_params(const resa_params_t* p) {
  if (p == nullptr) return RESA_ERR_INVALID_ARG;
  if (!(p->keep_ratio >= 0.0 && p->keep_ratio <= 1.0)) return RESA_ERR_INVALID_ARG;
  if (p->n_min_blocks < 0 || p->n_local_blocks < 0) return RESA_ERR_INVALID_ARG;
  if (!(p->sm_scale >= 0.f) || std::isinf(p->sm_scale)) return RESA_ERR_INVALID_ARG;
  return RESA_OK;
}

CacheView view(const resa_cache_t* c) {
  CacheView v;
  v.B = c->batch;
  v.Hq = c->num_q_heads;
  v.Hkv = c->num_kv_heads;
  v.g = c->num_q_heads / c->num_kv_heads;
  v.num_pages = c->num_pages;
  v.max_blocks = c->max_blocks_per_seq;
  v.k_pool = static_cast<uint16_t*>(c->k_pool);
  v.v_pool = static_cast<uint16_t*>(c->v_pool);
  v.page_table = c->page_table;
  v.seq_lens = c->seq_lens;
  v.summ = static_cast<uint16_t*>(c->summaries);
  v.status = c->device_status;
  v.active = nullptr;
  v.pending = 0;
  v.k_append = nullptr;
  v.v_append = nullptr;
  return v;
}

float scale_of(const resa_cache_t* c, const resa_params_t* p) {
  return p->sm_scale > 0.f ? p->sm_scale : 1.0f / std::sqrt(static_cast<float>(c->head_dim));
}

int64_t budget(int64_t M, const resa_params_t* p) {
  int64_t n = static_cast<int64_t>(std::ceil(static_cast<double>(M) * p->keep_ratio));
  if (n < p->n_min_blocks) n = p->n_min_blocks;
  if (n < p->n_local_blocks) n = p->n_local_blocks;
  if (n > M) n = M;
  return n;
}

resa_status_t auto_decode_splits(const resa_cache_t* c, int n_cap, int* out) {
  int sms = 0;
  const resa_status_t s = sm_count(&sms);
  if (s != RESA_OK) return s;
  // Algorithm 2's num_splits: as many splits as fit in one wave of resident
  // decode CTAs over batch * KV heads (no tail wave), with at least two
  // selected blocks per split. Fewer CTAs per SM are resident when the full
  // count would leave a split fewer than 16 selected blocks (measured: batch
  // 1 at 256K, 4 units of 820 blocks, runs its decode step faster with 38
  // splits of ~22 blocks than with 76 of ~11).
  const int units = c->batch * c->num_kv_heads;
  int per_sm = decode_ctas_per_sm();
  while (per_sm > 1 && n_cap < 16 * (sms * per_sm / units)) --per_sm;
  int splits = sms * per_sm / units;
  const int max_by_blocks = n_cap / 2 > 1 ? n_cap / 2 : 1;
  if (splits > max_by_blocks) splits = max_by_blocks;
  if (splits > 256) splits = 256;
  if (splits < 1) splits = 1;
  *out = splits;
  return RESA_OK;
}

resa_status_t auto_rectify_splits(const resa_cache_t* c, int f, int* out) {
  int sms = 0;
  const resa_status_t s = sm_count(&sms);
  if (s != RESA_OK) return s;
  const int units = c->batch * c->num_kv_heads * rectify_row_groups(c->num_q_heads / c->num_kv_heads, f);
  int splits = sms / units;
  const int64_t tiles = (static_cast<int64_t>(c->max_blocks_per_seq) * c->block_size + 63) / 64;
  if (splits > tiles) splits = static_cast<int>(tiles);
  if (splits > 256) splits = 256;
  if (splits < 1) splits = 1;
  *out = splits;
  return RESA_OK;
}

// Workspace regions; the calls run in stream order, so they alias.
size_t scores_bytes(const resa_cache_t* c) {
  return align_up(static_cast<size_t>(c->batch) * c->num_kv_heads * c->max_blocks_per_seq * sizeof(float));
}
size_t partial_bytes(size_t rows, int splits) {
  return align_up(rows * splits * kHeadDimHost * sizeof(float)) + align_up(rows * splits * sizeof(float));
}

}  // namespace

cudaError_t ensure_smem_attr(const void* func, int bytes, int slot) {
  static std::atomic<uint32_t> done[kMaxDevices];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint32_t bit = 1u << slot;
  if (dev < kMaxDevices && (done[dev].load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  if (e == cudaSuccess && dev < kMaxDevices) done[dev].fetch_or(bit, std::memory_order_acq_rel);
  return e;
}

}  // namespace resa

using namespace resa;

extern "C" {

int32_t resa_abi_version(void) { return RESA_ABI_VERSION; }

const char* resa_status_string(resa_status_t s) {
  switch (s) {
    case RESA_OK: return "RESA_OK";
    case RESA_ERR_INVALID_ARG: return "RESA_ERR_INVALID_ARG";
    case RESA_ERR_UNSUPPORTED: return "RESA_ERR_UNSUPPORTED";
    case RESA_ERR_WORKSPACE: return "RESA_ERR_WORKSPACE";
    case RESA_ERR_CUDA: return "RESA_ERR_CUDA";
    case RESA_ERR_DEVICE: return "RESA_ERR_DEVICE";
  }
  return "RESA_ERR_UNKNOWN";
}

resa_status_t resa_set_decode_wait_polls(uint32_t polls) {
  g_decode_wait_polls.store(polls, std::memory_order_relaxed);
  return RESA_OK;
}

resa_status_t resa_max_selected(const resa_cache_t* cache, const resa_params_t* params, int32_t* n_out) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if ((s = check_params(params)) != RESA_OK) return s;
  if (n_out == nullptr) return RESA_ERR_INVALID_ARG;
  *n_out = static_cast<int32_t>(budget(cache->max_blocks_per_seq, params));
  return RESA_OK;
}

resa_status_t resa_decode_num_splits(const resa_cache_t* cache, int32_t n_cap, int32_t* splits_out) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if (n_cap <= 0 || splits_out == nullptr) return RESA_ERR_INVALID_ARG;
  int v = 0;
  if ((s = auto_decode_splits(cache, n_cap, &v)) != RESA_OK) return s;
  *splits_out = v;
  return RESA_OK;
}

resa_status_t resa_rectify_num_splits(const resa_cache_t* cache, int32_t f, int32_t* splits_out) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if (f <= 0 || f > cache->max_blocks_per_seq * cache->block_size || splits_out == nullptr)
    return RESA_ERR_INVALID_ARG;
  int v = 0;
  if ((s = auto_rectify_splits(cache, f, &v)) != RESA_OK) return s;
  *splits_out = v;
  return RESA_OK;
}

resa_status_t resa_workspace_size(const resa_cache_t* cache, int32_t n_cap, int32_t num_splits, int32_t max_f,
                                  size_t* bytes_out) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if (n_cap <= 0 || num_splits < 0 || max_f < 0 || bytes_out == nullptr) return RESA_ERR_INVALID_ARG;
  int ds = num_splits;
  if (ds == 0 && (s = auto_decode_splits(cache, n_cap, &ds)) != RESA_OK) return s;
  size_t need = scores_bytes(cache);
  const size_t dec = partial_bytes(static_cast<size_t>(cache->batch) * cache->num_q_heads, ds);
  if (dec > need) need = dec;
  if (max_f > 0) {
    int rs = 0;
    if ((s = auto_rectify_splits(cache, max_f, &rs)) != RESA_OK) return s;
    // fewer rows or more splits never need more than the largest f's layout
    int rs1 = 0;
    if ((s = auto_rectify_splits(cache, 1, &rs1)) != RESA_OK) return s;
    const size_t rows = static_cast<size_t>(cache->batch) * max_f * cache->num_q_heads;
    const size_t rect = partial_bytes(rows, rs > rs1 ? rs : rs1);
    if (rect > need) need = rect;
  }
  *bytes_out = need;
  return RESA_OK;
}

resa_status_t resa_update_summaries(const resa_cache_t* cache, int32_t block_begin, int32_t block_end,
                                    void* stream) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if (block_begin < 0 || block_begin > cache->max_blocks_per_seq) return RESA_ERR_INVALID_ARG;
  if (block_end != -1 && (block_end < block_begin || block_end > cache->max_blocks_per_seq))
    return RESA_ERR_INVALID_ARG;
  const cudaError_t e =
      launch_update_summaries(view(cache), block_begin, block_end, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? RESA_OK : RESA_ERR_CUDA;
}

resa_status_t resa_commit_kv_active(const resa_cache_t* cache, const int32_t* active, const void* k_new,
                                    const void* v_new, int32_t n_tokens, int32_t overwrite, void* stream) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if (n_tokens < 0 || n_tokens > cache->max_blocks_per_seq * cache->block_size) return RESA_ERR_INVALID_ARG;
  if (overwrite != 0 && overwrite != 1) return RESA_ERR_INVALID_ARG;
  if (n_tokens > 0 && (k_new == nullptr || v_new == nullptr)) return RESA_ERR_INVALID_ARG;
  if (n_tokens > 0 && (!aligned16(k_new) || !aligned16(v_new))) return RESA_ERR_INVALID_ARG;
  CacheView v = view(cache);
  v.active = active;
  const cudaError_t e = launch_commit(v, static_cast<const uint16_t*>(k_new), static_cast<const uint16_t*>(v_new),
                                      n_tokens, overwrite == 1, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? RESA_OK : RESA_ERR_CUDA;
}

resa_status_t resa_commit_kv(const resa_cache_t* cache, const void* k_new, const void* v_new, int32_t n_tokens,
                             int32_t overwrite, void* stream) {
  return resa_commit_kv_active(cache, nullptr, k_new, v_new, n_tokens, overwrite, stream);
}

resa_status_t resa_select_blocks(const resa_cache_t* cache, const void* q, const resa_params_t* params,
                                 int32_t* indices, int32_t* counts, int32_t n_cap, void* workspace,
                                 size_t workspace_bytes, void* stream) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if ((s = check_params(params)) != RESA_OK) return s;
  if (q == nullptr || indices == nullptr || counts == nullptr || n_cap <= 0) return RESA_ERR_INVALID_ARG;
  if (!aligned16(q)) return RESA_ERR_INVALID_ARG;
  if (workspace == nullptr || workspace_bytes < scores_bytes(cache)) return RESA_ERR_WORKSPACE;
  int sms = 0;
  if ((s = sm_count(&sms)) != RESA_OK) return s;
  const cudaError_t e = launch_select(view(cache), static_cast<const uint16_t*>(q), params->keep_ratio,
                                      params->n_min_blocks, params->n_local_blocks, indices, counts, n_cap,
                                      static_cast<float*>(workspace), sms, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? RESA_OK : RESA_ERR_CUDA;
}

resa_status_t resa_sparse_decode(const resa_cache_t* cache, const void* q, const int32_t* indices,
                                 const int32_t* counts, int32_t n_cap, const resa_params_t* params, void* out,
                                 float* lse, int32_t num_splits, void* workspace, size_t workspace_bytes,
                                 void* stream) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if ((s = check_params(params)) != RESA_OK) return s;
  if (q == nullptr || indices == nullptr || counts == nullptr || out == nullptr || n_cap <= 0 || num_splits < 0)
    return RESA_ERR_INVALID_ARG;
  if (!aligned16(q)) return RESA_ERR_INVALID_ARG;
  int splits = num_splits;
  if (splits == 0 && (s = auto_decode_splits(cache, n_cap, &splits)) != RESA_OK) return s;
  if (splits > 1024) return RESA_ERR_INVALID_ARG;
  const size_t rows = static_cast<size_t>(cache->batch) * cache->num_q_heads;
  if (workspace == nullptr || workspace_bytes < partial_bytes(rows, splits)) return RESA_ERR_WORKSPACE;
  CUtensorMap tk, tv;
  if ((s = pool_tensor_map(cache, cache->k_pool, &tk)) != RESA_OK) return s;
  if ((s = pool_tensor_map(cache, cache->v_pool, &tv)) != RESA_OK) return s;
  float* o_part = static_cast<float*>(workspace);
  float* lse_part = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                             align_up(rows * splits * kHeadDimHost * sizeof(float)));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = launch_sparse_decode(view(cache), tk, tv, static_cast<const uint16_t*>(q), indices, counts, n_cap,
                                       scale_of(cache, params), splits, o_part, lse_part, st,
                                       g_decode_wait_polls.load(std::memory_order_relaxed));
  if (e == cudaSuccess)
    e = launch_merge(o_part, lse_part, static_cast<int>(rows), splits, static_cast<uint16_t*>(out), lse, st);
  return e == cudaSuccess ? RESA_OK : RESA_ERR_CUDA;
}

resa_status_t resa_decode_step(const resa_cache_t* cache, const void* k_new, const void* v_new, const void* q,
                               const resa_params_t* params, int32_t* indices, int32_t* counts, int32_t n_cap,
                               void* out, float* lse, int32_t num_splits, void* workspace, size_t workspace_bytes,
                               void* stream) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if ((s = check_params(params)) != RESA_OK) return s;
  if (k_new == nullptr || v_new == nullptr || q == nullptr || indices == nullptr || counts == nullptr ||
      out == nullptr || n_cap <= 0 || num_splits < 0)
    return RESA_ERR_INVALID_ARG;
  if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(q)) return RESA_ERR_INVALID_ARG;
  int splits = num_splits;
  if (splits == 0 && (s = auto_decode_splits(cache, n_cap, &splits)) != RESA_OK) return s;
  if (splits > 1024) return RESA_ERR_INVALID_ARG;
  const size_t rows = static_cast<size_t>(cache->batch) * cache->num_q_heads;
  if (workspace == nullptr || workspace_bytes < scores_bytes(cache) ||
      workspace_bytes < partial_bytes(rows, splits))
    return RESA_ERR_WORKSPACE;
  int sms = 0;
  if ((s = sm_count(&sms)) != RESA_OK) return s;
  CUtensorMap tk, tv;
  if ((s = pool_tensor_map(cache, cache->k_pool, &tk)) != RESA_OK) return s;
  if ((s = pool_tensor_map(cache, cache->v_pool, &tv)) != RESA_OK) return s;
  CacheView v = view(cache);
  v.pending = 1;
  v.k_append = static_cast<const uint16_t*>(k_new);
  v.v_append = static_cast<const uint16_t*>(v_new);
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  // scores and partials alias: the partials are written after the top-n has read the scores
  cudaError_t e = launch_select(v, static_cast<const uint16_t*>(q), params->keep_ratio, params->n_min_blocks,
                                params->n_local_blocks, indices, counts, n_cap, static_cast<float*>(workspace), sms,
                                st);
  float* o_part = static_cast<float*>(workspace);
  float* lse_part = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                             align_up(rows * splits * kHeadDimHost * sizeof(float)));
  if (e == cudaSuccess)
    e = launch_sparse_decode(v, tk, tv, static_cast<const uint16_t*>(q), indices, counts, n_cap,
                             scale_of(cache, params), splits, o_part, lse_part, st,
                                       g_decode_wait_polls.load(std::memory_order_relaxed));
  if (e == cudaSuccess)
    e = launch_merge(o_part, lse_part, static_cast<int>(rows), splits, static_cast<uint16_t*>(out), lse, st, nullptr,
                     cache->num_q_heads, &v);
  return e == cudaSuccess ? RESA_OK : RESA_ERR_CUDA;
}

resa_status_t resa_rectify_attention_active(const resa_cache_t* cache, const int32_t* active, const void* q_new,
                                            const void* k_new, const void* v_new, int32_t f,
                                            const resa_params_t* params, void* out, float* lse, void* workspace,
                                            size_t workspace_bytes, void* stream) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if ((s = check_params(params)) != RESA_OK) return s;
  if (q_new == nullptr || k_new == nullptr || v_new == nullptr || out == nullptr) return RESA_ERR_INVALID_ARG;
  if (f <= 0 || f > cache->max_blocks_per_seq * cache->block_size) return RESA_ERR_INVALID_ARG;
  if (!aligned16(q_new) || !aligned16(k_new) || !aligned16(v_new)) return RESA_ERR_INVALID_ARG;
  int splits = 0;
  if ((s = auto_rectify_splits(cache, f, &splits)) != RESA_OK) return s;
  const size_t rows = static_cast<size_t>(cache->batch) * f * cache->num_q_heads;
  if (workspace == nullptr || workspace_bytes < partial_bytes(rows, splits)) return RESA_ERR_WORKSPACE;
  CUtensorMap tk, tv;
  if ((s = pool_tensor_map(cache, cache->k_pool, &tk)) != RESA_OK) return s;
  if ((s = pool_tensor_map(cache, cache->v_pool, &tv)) != RESA_OK) return s;
  float* o_part = static_cast<float*>(workspace);
  float* lse_part = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                             align_up(rows * splits * kHeadDimHost * sizeof(float)));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  CUtensorMap tkn, tvn;
  if ((s = new_kv_tensor_map(cache, k_new, f, &tkn)) != RESA_OK) return s;
  if ((s = new_kv_tensor_map(cache, v_new, f, &tvn)) != RESA_OK) return s;
  CacheView v = view(cache);
  v.active = active;
  cudaError_t e = launch_rectify(v, tk, tv, tkn, tvn, static_cast<const uint16_t*>(q_new),
                                 static_cast<const uint16_t*>(k_new), static_cast<const uint16_t*>(v_new), f,
                                 scale_of(cache, params), splits, o_part, lse_part, st);
  if (e == cudaSuccess)
    e = launch_merge(o_part, lse_part, static_cast<int>(rows), splits, static_cast<uint16_t*>(out), lse, st, active,
                     f * cache->num_q_heads);
  return e == cudaSuccess ? RESA_OK : RESA_ERR_CUDA;
}

resa_status_t resa_rectify_attention(const resa_cache_t* cache, const void* q_new, const void* k_new,
                                     const void* v_new, int32_t f, const resa_params_t* params, void* out,
                                     float* lse, void* workspace, size_t workspace_bytes, void* stream) {
  return resa_rectify_attention_active(cache, nullptr, q_new, k_new, v_new, f, params, out, lse, workspace,
                                       workspace_bytes, stream);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Static scratch for resa_sparse_decode_static (callers that cannot allocate).
// In host code `g_static_scratch` names a host-side stand-in, not the device
// buffer, so its device address is looked up once per device with
// cudaGetSymbolAddress (that device current) and passed to the kernels.
// ---------------------------------------------------------------------------
static __device__ __align__(256) unsigned char g_static_scratch[RESA_STATIC_SCRATCH_BYTES];

namespace {
std::mutex g_static_mu;
void* g_static_ptr[resa::kMaxDevices];

resa_status_t static_scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return RESA_ERR_CUDA;
  if (dev >= resa::kMaxDevices) return RESA_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (g_static_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr) return RESA_ERR_CUDA;
    g_static_ptr[dev] = p;
  }
  *out = g_static_ptr[dev];
  return RESA_OK;
}
}  // namespace

extern "C" {

resa_status_t resa_sparse_decode_static(const resa_cache_t* cache, const void* q, const int32_t* indices,
                                        const int32_t* counts, int32_t n_cap, const resa_params_t* params,
                                        void* out, float* lse, int32_t num_splits, void* stream) {
  resa_status_t s = check_cache(cache);
  if (s != RESA_OK) return s;
  if ((s = check_params(params)) != RESA_OK) return s;
  if (q == nullptr || indices == nullptr || counts == nullptr || out == nullptr || n_cap <= 0 || num_splits < 0)
    return RESA_ERR_INVALID_ARG;
  if (!aligned16(q)) return RESA_ERR_INVALID_ARG;
  int splits = num_splits;
  if (splits == 0 && (s = auto_decode_splits(cache, n_cap, &splits)) != RESA_OK) return s;
  if (splits > 1024) return RESA_ERR_INVALID_ARG;
  const size_t rows = static_cast<size_t>(cache->batch) * cache->num_q_heads;
  if (partial_bytes(rows, splits) > RESA_STATIC_SCRATCH_BYTES) return RESA_ERR_WORKSPACE;
  void* scratch = nullptr;
  if ((s = static_scratch_address(&scratch)) != RESA_OK) return s;
  CUtensorMap tk, tv;
  if ((s = pool_tensor_map(cache, cache->k_pool, &tk)) != RESA_OK) return s;
  if ((s = pool_tensor_map(cache, cache->v_pool, &tv)) != RESA_OK) return s;
  float* o_part = static_cast<float*>(scratch);
  float* lse_part = reinterpret_cast<float*>(static_cast<char*>(scratch) +
                                             align_up(rows * splits * kHeadDimHost * sizeof(float)));
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t e = launch_sparse_decode(view(cache), tk, tv, static_cast<const uint16_t*>(q), indices, counts, n_cap,
                                       scale_of(cache, params), splits, o_part, lse_part, st,
                                       g_decode_wait_polls.load(std::memory_order_relaxed));
  if (e == cudaSuccess)
    e = launch_merge(o_part, lse_part, static_cast<int>(rows), splits, static_cast<uint16_t*>(out), lse, st);
  return e == cudaSuccess ? RESA_OK : RESA_ERR_CUDA;
}

resa_status_t resa_read_device_error(const resa_cache_t* cache, int32_t* code_out, int32_t* detail_out,
                                     void* stream) {
  if (cache == nullptr || cache->device_status == nullptr) return RESA_ERR_INVALID_ARG;
  const cudaStream_t st = static_cast<cudaStream_t>(stream);
  int32_t h[2] = {0, 0};
  if (cudaMemcpyAsync(h, cache->device_status, sizeof(h), cudaMemcpyDeviceToHost, st) != cudaSuccess)
    return RESA_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return RESA_ERR_CUDA;
  if (h[0] != 0 && cudaMemsetAsync(cache->device_status, 0, 2 * sizeof(int32_t), st) != cudaSuccess)
    return RESA_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return RESA_ERR_CUDA;
  if (code_out != nullptr) *code_out = h[0];
  if (detail_out != nullptr) *detail_out = h[1];
  return h[0] != 0 ? RESA_ERR_DEVICE : RESA_OK;
}

}  // extern "C"
