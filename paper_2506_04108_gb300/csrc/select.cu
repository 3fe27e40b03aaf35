// Block selection (Section 2.1 "Block Selection"; Eq. 4 and Eq. 5).
//
// score_kernel  grid (block chunks, KV head, sequence). Each CTA forms the
//               pooled query of its GQA group (mean of the g heads, fp32) and
//               scores 64 blocks: a half-warp takes one block, each lane one
//               16-byte chunk (8 dims) of k_min and k_max, so a warp reads two
//               contiguous 512-byte summaries per load instruction. The
//               128-dim sum is a fixed-order butterfly over the 16 lanes.
// topn_kernel   grid (KV head, sequence), 1024 threads. The n of Eq. 5 is
//               evaluated on the device from the device-resident length. The
//               n-th largest order-preserving key is found by an 8-bit radix
//               select (4 histogram passes over keys staged in shared
//               memory, warp-aggregated atomics), then the selected ids are
//               written in ascending order by a ballot compaction that also
//               resolves ties at the threshold toward the lower block index.
//               The last n_local blocks carry the maximum key (score +inf).
#include "resa_device.cuh"
#include "resa_launch.h"

namespace resa {
namespace {

constexpr int kScoreWarps = 8;
constexpr int kScoreUnroll = 4;                                    // 2 blocks per warp per step
constexpr int kBlocksPerScoreCta = kScoreWarps * 2 * kScoreUnroll;  // 64
constexpr int kTopnThreads = 1024;
constexpr int kTopnWarps = kTopnThreads / 32;
constexpr int kKeysInSmem = 32768;                                 // 128 KB of staged keys

__device__ __forceinline__ float quest_term8(const float* q, const uint4& mn, const uint4& mx) {
  const uint32_t a[4] = {mn.x, mn.y, mn.z, mn.w};
  const uint32_t c[4] = {mx.x, mx.y, mx.z, mx.w};
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    s += fmaxf(q[2 * i] * bf16_lo(c[i]), q[2 * i] * bf16_lo(a[i]));
    s += fmaxf(q[2 * i + 1] * bf16_hi(c[i]), q[2 * i + 1] * bf16_hi(a[i]));
  }
  return s;
}

__global__ void __launch_bounds__(256) score_kernel(CacheView c, const uint16_t* __restrict__ q,
                                                    float* __restrict__ scores) {
  const int b = blockIdx.z, h = blockIdx.y;
  const int T = c.seq_lens[b];
  if (T < 0 || T > c.max_blocks * kBlock) return;  // reported by topn_kernel
  const int M = (T + kBlock - 1) / kBlock;
  const int base = blockIdx.x * kBlocksPerScoreCta;
  if (base >= M) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ch = lane & 15, half = lane >> 4;

  // pooled query (mean of the group's heads) for this lane's 8 dims
  float qp[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) qp[j] = 0.f;
  const uint16_t* qg = q + (static_cast<size_t>(b) * c.Hq + h * c.g) * kHeadDim + ch * 8;
  for (int i = 0; i < c.g; ++i) {
    const uint4 v = *reinterpret_cast<const uint4*>(qg + i * kHeadDim);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      qp[2 * j] += bf16_lo(w[j]);
      qp[2 * j + 1] += bf16_hi(w[j]);
    }
  }
  const float inv_g = 1.0f / static_cast<float>(c.g);
#pragma unroll
  for (int j = 0; j < 8; ++j) qp[j] = qp[j] * inv_g;

  const uint16_t* sb = c.summ + (static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks * 2 * kHeadDim;
  uint4 mn[kScoreUnroll], mx[kScoreUnroll];
  int blk[kScoreUnroll];
#pragma unroll
  for (int u = 0; u < kScoreUnroll; ++u) {
    blk[u] = base + warp * (2 * kScoreUnroll) + 2 * u + half;
    if (blk[u] < M) {
      const uint16_t* s = sb + static_cast<size_t>(blk[u]) * 2 * kHeadDim + ch * 8;
      mn[u] = *reinterpret_cast<const uint4*>(s);
      mx[u] = *reinterpret_cast<const uint4*>(s + kHeadDim);
    } else {
      mn[u] = make_uint4(0, 0, 0, 0);
      mx[u] = make_uint4(0, 0, 0, 0);
    }
  }
  float* out = scores + (static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks;
#pragma unroll
  for (int u = 0; u < kScoreUnroll; ++u) {
    float s = quest_term8(qp, mn[u], mx[u]);
    s += __shfl_xor_sync(0xffffffffu, s, 8);
    s += __shfl_xor_sync(0xffffffffu, s, 4);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    if (ch == 0 && blk[u] < M) out[blk[u]] = s;
  }
}

// Order-preserving map of an fp32 score to uint32 (larger score, larger key).
__device__ __forceinline__ uint32_t score_key(float s) {
  const uint32_t u = __float_as_uint(s);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive scan of one value per warp (kTopnWarps values) by warp 0.
__device__ __forceinline__ void scan_warp_totals(int* vals, int* total) {
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < 32) {
    const int v = vals[lane];
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    vals[lane] = x - v;
    if (lane == 31) *total = x;
  }
}

__global__ void __launch_bounds__(kTopnThreads) topn_kernel(CacheView c, const float* __restrict__ scores,
                                                            double keep, int n_min, int n_local,
                                                            int32_t* __restrict__ indices,
                                                            int32_t* __restrict__ counts, int n_cap) {
  extern __shared__ uint32_t keys_smem[];
  __shared__ int hist[256];
  __shared__ int warp_a[kTopnWarps], warp_b[kTopnWarps];
  __shared__ int sh_digit, sh_rem, sh_tot;

  const int b = blockIdx.y, h = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int32_t* out = indices + (static_cast<size_t>(b) * c.Hkv + h) * n_cap;
  const int T = c.seq_lens[b];
  if (T < 0 || T > c.max_blocks * kBlock) {
    if (tid == 0) {
      record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
      counts[b * c.Hkv + h] = 0;
    }
    for (int i = tid; i < n_cap; i += kTopnThreads) out[i] = -1;
    return;
  }
  const int M = (T + kBlock - 1) / kBlock;
  // Eq. 5 on the device: n = max(n_min, ceil(M * keep)), n_local <= n <= M
  long long nn = static_cast<long long>(ceil(static_cast<double>(M) * keep));
  nn = max(nn, static_cast<long long>(n_min));
  nn = max(nn, static_cast<long long>(n_local));
  nn = min(nn, static_cast<long long>(M));
  int n = static_cast<int>(nn);
  if (n > n_cap) {
    if (tid == 0) record_error(c.status, RESA_DEV_BUDGET_OVER_CAP, b * c.Hkv + h);
    n = n_cap;
  }
  const float* sc = scores + (static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks;
  const int first_forced = M - n_local;
  const bool staged = c.max_blocks <= kKeysInSmem;  // the host sized the buffer from max_blocks
  if (staged) {
    for (int i = tid; i < M; i += kTopnThreads)
      keys_smem[i] = (i >= first_forced) ? 0xFFFFFFFFu : score_key(sc[i]);
  }
  __syncthreads();
  auto key_of = [&](int i) -> uint32_t {
    if (staged) return keys_smem[i];
    return (i >= first_forced) ? 0xFFFFFFFFu : score_key(sc[i]);
  };
  const int M_round = ((M + kTopnThreads - 1) / kTopnThreads) * kTopnThreads;

  // ---- radix select of the n-th largest key ----
  uint32_t prefix = 0, pmask = 0;
  int rem = n;
  if (n > 0) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      if (tid < 256) hist[tid] = 0;
      __syncthreads();
      for (int i = tid; i < M_round; i += kTopnThreads) {
        uint32_t d = 0x100u;  // sentinel: not counted
        if (i < M) {
          const uint32_t k = key_of(i);
          if ((k & pmask) == prefix) d = (k >> shift) & 0xFFu;
        }
        const unsigned peers = __match_any_sync(0xffffffffu, d);
        if (d != 0x100u && lane == __ffs(peers) - 1) atomicAdd(&hist[d], __popc(peers));
      }
      __syncthreads();
      if (warp == 0) {
        // lane l owns digits 255-8l ... 248-8l (descending)
        int cnt[8], sum = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          cnt[j] = hist[255 - 8 * lane - j];
          sum += cnt[j];
        }
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        const int excl = incl - sum;
        if (excl < rem && rem <= incl) {
          int cum = excl;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (cum + cnt[j] >= rem) {
              sh_digit = 255 - 8 * lane - j;
              sh_rem = rem - cum;
              break;
            }
            cum += cnt[j];
          }
        }
      }
      __syncthreads();
      prefix |= static_cast<uint32_t>(sh_digit) << shift;
      pmask |= 0xFFu << shift;
      rem = sh_rem;
    }
  }
  // keys > prefix are all taken; of the keys == prefix, the `rem` lowest ids.
  const uint32_t tau = prefix;
  const int take_eq = (n > 0) ? rem : 0;

  // ---- ordered compaction: each warp owns a contiguous id range ----
  const int per_warp = ((M + kTopnWarps * 32 - 1) / (kTopnWarps * 32)) * 32;
  const int w0 = warp * per_warp, w1 = min(M, w0 + per_warp);
  int gt = 0, eq = 0;
  if (n > 0) {
    for (int i0 = w0; i0 < w0 + per_warp; i0 += 32) {
      const int i = i0 + lane;
      const uint32_t k = (i < w1) ? key_of(i) : 0u;
      const bool in = i < w1;
      gt += __popc(__ballot_sync(0xffffffffu, in && k > tau));
      eq += __popc(__ballot_sync(0xffffffffu, in && k == tau));
    }
  }
  if (lane == 0) {
    warp_a[warp] = eq;
    warp_b[warp] = gt;
  }
  __syncthreads();
  scan_warp_totals(warp_a, &sh_tot);  // exclusive prefix of equal keys per warp
  __syncthreads();
  if (lane == 0) {
    const int eq_before = warp_a[warp];
    const int eq_taken = max(0, min(eq, take_eq - eq_before));
    warp_b[warp] = gt + eq_taken;
  }
  __syncthreads();
  scan_warp_totals(warp_b, &sh_tot);  // exclusive prefix of selected ids per warp
  __syncthreads();
  if (n > 0) {
    int eq_seen = warp_a[warp];
    int pos = warp_b[warp];
    for (int i0 = w0; i0 < w0 + per_warp; i0 += 32) {
      const int i = i0 + lane;
      const bool in = i < w1;
      const uint32_t k = in ? key_of(i) : 0u;
      const bool is_eq = in && k == tau;
      const unsigned eqm = __ballot_sync(0xffffffffu, is_eq);
      const int my_eq_rank = eq_seen + __popc(eqm & ((1u << lane) - 1u));
      const bool sel = in && (k > tau || (is_eq && my_eq_rank < take_eq));
      const unsigned selm = __ballot_sync(0xffffffffu, sel);
      if (sel) out[pos + __popc(selm & ((1u << lane) - 1u))] = i;
      eq_seen += __popc(eqm);
      pos += __popc(selm);
    }
  }
  for (int i = n + tid; i < n_cap; i += kTopnThreads) out[i] = -1;
  if (tid == 0) counts[b * c.Hkv + h] = n;
}

}  // namespace

size_t select_smem_bytes(int max_blocks) {
  const int staged = max_blocks <= kKeysInSmem ? max_blocks : 0;
  return static_cast<size_t>(staged) * sizeof(uint32_t);
}

cudaError_t launch_select(const CacheView& c, const uint16_t* q, double keep, int n_min, int n_local,
                          int32_t* indices, int32_t* counts, int n_cap, float* scores, cudaStream_t st) {
  const dim3 sgrid((c.max_blocks + kBlocksPerScoreCta - 1) / kBlocksPerScoreCta, c.Hkv, c.B);
  score_kernel<<<sgrid, kScoreWarps * 32, 0, st>>>(c, q, scores);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t smem = select_smem_bytes(c.max_blocks);
  if (smem > 48 * 1024) {
    // sized for the largest staging buffer so one attribute call serves every cache
    e = ensure_smem_attr(reinterpret_cast<const void*>(topn_kernel), select_smem_bytes(kKeysInSmem), 2);
    if (e != cudaSuccess) return e;
  }
  topn_kernel<<<dim3(c.Hkv, c.B), kTopnThreads, smem, st>>>(c, scores, keep, n_min, n_local, indices, counts,
                                                            n_cap);
  return cudaGetLastError();
}

}  // namespace resa
