// Internal launcher interface between the C-ABI layer (resa_api.cu) and the
// kernel translation units. Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "resa.h"

namespace resa {

constexpr int kHeadDimHost = 128;  // supported head_dim
constexpr int kBlockHost = 16;     // supported block_size (paper's b)

// Plain-old-data view of resa_cache_t handed to kernels by value.
struct CacheView {
  int B, Hq, Hkv, g;
  int num_pages, max_blocks;
  uint16_t* k_pool;
  uint16_t* v_pool;
  const int32_t* page_table;
  int32_t* seq_lens;
  uint16_t* summ;
  int32_t* status;
  const int32_t* active;  // [B]: sequences with 0 are left out of commits and rectification; null = all
  // Fused decode step: `pending` tokens (0 or 1) are appended by the running
  // call and not yet counted in seq_lens, which its last kernel advances;
  // every kernel of the call works on T = seq_lens[b] + pending. The appended
  // key and value are k_append / v_append, bf16 [B][Hkv][128].
  int pending;
  const uint16_t* k_append;
  const uint16_t* v_append;
};

#ifdef __CUDACC__
// Element offsets into the paged pool and the block summaries.
__device__ __forceinline__ size_t pool_off(const CacheView& c, int page, int h, int row) {
  return ((static_cast<size_t>(page) * c.Hkv + h) * 16 + row) * 128;
}
__device__ __forceinline__ size_t summ_off(const CacheView& c, int b, int h, int blk) {
  return ((static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks + blk) * 2 * 128;
}
#endif

// Launches `kernel` with programmatic stream serialization (see
// pdl_launch_dependents / pdl_wait in resa_device.cuh).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Sets cudaFuncAttributeMaxDynamicSharedMemorySize of `func` once per device
// (kernel-launch paths then make no attribute calls, e.g. under graph capture).
cudaError_t ensure_smem_attr(const void* func, int bytes, int slot);

// kv_commit.cu
cudaError_t launch_commit(const CacheView& c, const uint16_t* k_new, const uint16_t* v_new, int n_tokens,
                          bool overwrite, cudaStream_t st);
cudaError_t launch_update_summaries(const CacheView& c, int block_begin, int block_end, cudaStream_t st);

// select.cu
size_t select_smem_bytes(int max_blocks);
int select_max_blocks();  // largest max_blocks_per_seq the selection supports
cudaError_t launch_select(const CacheView& c, const uint16_t* q, double keep, int n_min, int n_local,
                          int32_t* indices, int32_t* counts, int n_cap, float* scores, int sm_count,
                          cudaStream_t st);

// sparse_decode.cu
int decode_ctas_per_sm();  // resident decode CTAs per SM (occupancy), >= 1
// `wait_polls`: polls of one copy's barrier before a warp gives up
// (RESA_DEV_WAIT_TIMEOUT); copies already issued are then still awaited with
// the default limit before the CTA exits.
cudaError_t launch_sparse_decode(const CacheView& c, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                                 const uint16_t* q, const int32_t* indices, const int32_t* counts, int n_cap,
                                 float sm_scale, int splits, float* o_part, float* lse_part, cudaStream_t st,
                                 uint32_t wait_polls);
// `advance` (a fused decode step's view, pending > 0): the merge also counts
// the appended token in seq_lens; rows_per_seq must then be Hq.
cudaError_t launch_merge(const float* o_part, const float* lse_part, int rows, int splits, uint16_t* out,
                         float* lse_out, cudaStream_t st, const int32_t* active = nullptr, int rows_per_seq = 1,
                         const CacheView* advance = nullptr);

// rectify.cu
int rectify_row_groups(int g, int f);
cudaError_t launch_rectify(const CacheView& c, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                           const CUtensorMap& tm_kn, const CUtensorMap& tm_vn, const uint16_t* q_new,
                           const uint16_t* k_new, const uint16_t* v_new, int f, float sm_scale, int splits,
                           float* o_part, float* lse_part, cudaStream_t st);

}  // namespace resa
