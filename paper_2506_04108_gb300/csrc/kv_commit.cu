// KV commit and block-summary kernels (Algorithm 1 cache updates; Eq. 3).
//
//  * append:    one CTA per sequence writes the new tokens into their pages,
//               folds them into the touched blocks' min/max (the online update
//               of Section 2.1; min/max of bf16 values is exact, so this equals
//               a recompute), and finally advances seq_lens[b]. Keeping a
//               sequence inside one CTA lets the same kernel read and advance
//               the device-resident length without a second launch.
//  * overwrite: grid (touched block, sequence); each CTA writes the dense K/V
//               of its block and recomputes the block's summary from all of
//               its valid keys (a min/max cannot be "un-applied").
//  * bulk:      one warp per block recomputes Eq. 3 from the paged keys.
// A NaN in a valid key makes that dimension of its block's min and max NaN.
#include "resa_device.cuh"
#include "resa_launch.h"

namespace resa {
namespace {

__global__ void __launch_bounds__(256) commit_append_kernel(CacheView c, const uint16_t* __restrict__ k_new,
                                                            const uint16_t* __restrict__ v_new, int n) {
  pdl_wait();  // no early launch of dependents: they may read the summaries and lengths written here
  const int b = blockIdx.x;
  if (c.active != nullptr && c.active[b] == 0) return;
  const int T = c.seq_lens[b];
  const int cap = c.max_blocks * kBlock;
  if (T < 0 || T > cap - n) {
    if (threadIdx.x == 0) record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
    return;
  }
  const int H = c.Hkv;
  // 1. the new tokens, 16 bytes per thread-item
  const int items = n * H * 16;
  for (int it = threadIdx.x; it < items; it += blockDim.x) {
    const int ch = it & 15, th = it >> 4, h = th % H, t = th / H;
    const int pos = T + t;
    const int page = c.page_table[static_cast<size_t>(b) * c.max_blocks + (pos >> 4)];
    if (page < 0 || page >= c.num_pages) {
      record_error(c.status, RESA_DEV_PAGE_RANGE, b);
      continue;
    }
    const size_t dst = pool_off(c, page, h, pos & 15) + ch * 8;
    const size_t src = ((static_cast<size_t>(b) * n + t) * H + h) * kHeadDim + ch * 8;
    *reinterpret_cast<uint4*>(c.k_pool + dst) = *reinterpret_cast<const uint4*>(k_new + src);
    *reinterpret_cast<uint4*>(c.v_pool + dst) = *reinterpret_cast<const uint4*>(v_new + src);
  }
  // 2. online min/max of the touched blocks (from the new keys + old summary)
  const int blk0 = T >> 4, nb = ((T + n - 1) >> 4) - blk0 + 1;
  const int sitems = (n > 0 ? nb : 0) * H * 16;
  for (int it = threadIdx.x; it < sitems; it += blockDim.x) {
    const int ch = it & 15, bh = it >> 4, h = bh % H, blk = blk0 + bh / H;
    float mn[8], mx[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      mn[j] = __int_as_float(0x7f800000);
      mx[j] = -__int_as_float(0x7f800000);
    }
    uint16_t* s = c.summ + summ_off(c, b, h, blk);
    if (blk * kBlock < T) {  // block already holds keys: start from its summary
      minmax8(*reinterpret_cast<const uint4*>(s + ch * 8), mn, mx);
      minmax8(*reinterpret_cast<const uint4*>(s + kHeadDim + ch * 8), mn, mx);
    }
    const int p_lo = max(blk * kBlock, T), p_hi = min(blk * kBlock + kBlock, T + n);
    for (int p = p_lo; p < p_hi; ++p) {
      const size_t src = ((static_cast<size_t>(b) * n + (p - T)) * H + h) * kHeadDim + ch * 8;
      minmax8(*reinterpret_cast<const uint4*>(k_new + src), mn, mx);
    }
    *reinterpret_cast<uint4*>(s + ch * 8) = to_bf16x8(mn);
    *reinterpret_cast<uint4*>(s + kHeadDim + ch * 8) = to_bf16x8(mx);
  }
  __syncthreads();
  if (threadIdx.x == 0) c.seq_lens[b] = T + n;
}

__global__ void __launch_bounds__(256) commit_overwrite_kernel(CacheView c, const uint16_t* __restrict__ k_new,
                                                               const uint16_t* __restrict__ v_new, int n) {
  pdl_wait();  // no early launch of dependents: they may read the summaries and lengths written here
  const int b = blockIdx.y;
  if (c.active != nullptr && c.active[b] == 0) return;
  const int T = c.seq_lens[b];
  const int cap = c.max_blocks * kBlock;
  if (T < n || T > cap) {
    if (threadIdx.x == 0 && blockIdx.x == 0) record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
    return;
  }
  const int start = T - n;
  const int blk = (start >> 4) + blockIdx.x;
  if (blk > ((T - 1) >> 4)) return;
  const int H = c.Hkv;
  const int page = c.page_table[static_cast<size_t>(b) * c.max_blocks + blk];
  if (page < 0 || page >= c.num_pages) {
    if (threadIdx.x == 0) record_error(c.status, RESA_DEV_PAGE_RANGE, b);
    return;
  }
  // 1. write the dense K/V of the tokens of this block
  const int p_lo = max(blk * kBlock, start), p_hi = min(blk * kBlock + kBlock, T);
  const int items = (p_hi - p_lo) * H * 16;
  for (int it = threadIdx.x; it < items; it += blockDim.x) {
    const int ch = it & 15, th = it >> 4, h = th % H, p = p_lo + th / H;
    const size_t dst = pool_off(c, page, h, p & 15) + ch * 8;
    const size_t src = ((static_cast<size_t>(b) * n + (p - start)) * H + h) * kHeadDim + ch * 8;
    *reinterpret_cast<uint4*>(c.k_pool + dst) = *reinterpret_cast<const uint4*>(k_new + src);
    *reinterpret_cast<uint4*>(c.v_pool + dst) = *reinterpret_cast<const uint4*>(v_new + src);
  }
  __syncthreads();  // this CTA's global writes are visible to its own threads after the barrier
  // 2. recompute Eq. 3 for this block from all its valid keys
  const int valid = min(kBlock, T - blk * kBlock);
  for (int it = threadIdx.x; it < H * 16; it += blockDim.x) {
    const int ch = it & 15, h = it >> 4;
    float mn[8], mx[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      mn[j] = __int_as_float(0x7f800000);
      mx[j] = -__int_as_float(0x7f800000);
    }
    const uint16_t* src = c.k_pool + pool_off(c, page, h, 0) + ch * 8;
    for (int r = 0; r < valid; ++r) minmax8(*reinterpret_cast<const uint4*>(src + r * kHeadDim), mn, mx);
    uint16_t* s = c.summ + summ_off(c, b, h, blk);
    *reinterpret_cast<uint4*>(s + ch * 8) = to_bf16x8(mn);
    *reinterpret_cast<uint4*>(s + kHeadDim + ch * 8) = to_bf16x8(mx);
  }
}

// One warp per (sequence, head, block): lanes 0-15 take rows 0-7, lanes 16-31
// rows 8-15, each lane one 16-byte chunk (8 dims); halves combine by shuffle.
__global__ void __launch_bounds__(256) update_summaries_kernel(CacheView c, int begin, int end) {
  pdl_wait();  // no early launch of dependents: they may read the summaries and lengths written here
  const int b = blockIdx.z, h = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int blk = begin + blockIdx.x * 8 + warp;
  const int T = c.seq_lens[b];
  if (T < 0 || T > c.max_blocks * kBlock) {
    if (threadIdx.x == 0 && blockIdx.x == 0 && h == 0) record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
    return;
  }
  const int M = (T + kBlock - 1) / kBlock;
  const int stop = end < 0 ? M : min(end, M);
  if (blk < begin || blk >= stop) return;
  const int page = c.page_table[static_cast<size_t>(b) * c.max_blocks + blk];
  if (page < 0 || page >= c.num_pages) {
    if (lane == 0) record_error(c.status, RESA_DEV_PAGE_RANGE, b);
    return;
  }
  const int valid = min(kBlock, T - blk * kBlock);
  const int ch = lane & 15, half = lane >> 4;
  float mn[8], mx[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    mn[j] = __int_as_float(0x7f800000);
    mx[j] = -__int_as_float(0x7f800000);
  }
  const uint16_t* src = c.k_pool + pool_off(c, page, h, 0) + ch * 8;
#pragma unroll
  for (int r = 0; r < 8; ++r) {
    const int row = half * 8 + r;
    if (row < valid) minmax8(*reinterpret_cast<const uint4*>(src + row * kHeadDim), mn, mx);
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    mn[j] = fmin_nan(mn[j], __shfl_xor_sync(0xffffffffu, mn[j], 16));
    mx[j] = fmax_nan(mx[j], __shfl_xor_sync(0xffffffffu, mx[j], 16));
  }
  uint16_t* s = c.summ + summ_off(c, b, h, blk);
  if (half == 0)
    *reinterpret_cast<uint4*>(s + ch * 8) = to_bf16x8(mn);
  else
    *reinterpret_cast<uint4*>(s + kHeadDim + ch * 8) = to_bf16x8(mx);
}

}  // namespace

cudaError_t launch_commit(const CacheView& c, const uint16_t* k_new, const uint16_t* v_new, int n, bool overwrite,
                          cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  if (!overwrite) return launch_pdl(commit_append_kernel, dim3(c.B), dim3(256), 0, st, c, k_new, v_new, n);
  const dim3 grid((n + kBlock - 1) / kBlock + 1, c.B);
  return launch_pdl(commit_overwrite_kernel, grid, dim3(256), 0, st, c, k_new, v_new, n);
}

cudaError_t launch_update_summaries(const CacheView& c, int begin, int end, cudaStream_t st) {
  const int last = end < 0 ? c.max_blocks : end;
  const int nblk = last - begin;
  if (nblk <= 0) return cudaSuccess;
  const dim3 grid((nblk + 7) / 8, c.Hkv, c.B);
  return launch_pdl(update_summaries_kernel, grid, dim3(256), 0, st, c, begin, end);
}

}  // namespace resa
