// Block selection (Section 2.1 "Block Selection"; Eq. 4 and Eq. 5).
//
// score_kernel  persistent, one CTA per SM: streams the block summaries in
//               32 KB chunks with bulk copies through a shared-memory ring and
//               scores them with the pooled query of the chunk's GQA group
//               (mean of the g heads, fp32); a half-warp takes one block, a
//               lane one 16-byte piece (8 dims) of k_min and k_max, and the
//               128-dim sum is a fixed-order butterfly over the 16 lanes.
// topn_kernel   one 8-CTA cluster per (sequence, KV head). The n of Eq. 5 is
//               evaluated on the device from the device-resident length. The
//               n-th largest order-preserving key is found by an 8-bit radix
//               select over keys staged in the CTAs' shared memory, with the
//               histograms summed across the cluster through distributed
//               shared memory; the selected ids are written in ascending order
//               by a ballot compaction that resolves ties at the threshold
//               toward the lower block index. The last n_local blocks carry
//               the maximum key (score +inf).
#include <cooperative_groups.h>

#include <atomic>

#include "resa_device.cuh"
#include "resa_launch.h"

namespace resa {
namespace {

constexpr int kScoreWarps = 8;
constexpr int kTopnCluster = 8;                                   // CTAs per (sequence, KV head)
constexpr int kTopnThreads = 256;
constexpr int kTopnWarps = kTopnThreads / 32;
constexpr int kTopnSmemMax = 200 * 1024;                           // staged keys per CTA, bytes

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

// Persistent score kernel: one CTA per SM. The (sequence, KV head) units'
// summaries are cut into chunks of 64 blocks (32 KB, contiguous); CTA x owns
// the chunk range [x * per, (x + 1) * per) of the flattened chunk list.
// Thread 0 streams the chunks with 1-D bulk copies into a kScoreStages-deep
// shared-memory ring; the 8 warps score each chunk from shared memory (a
// half-warp per block, a lane per 16-byte piece of k_min and k_max, fixed
// order 16-lane reduction) and release the stage.
constexpr int kScoreStages = 6;
constexpr int kMaxBatch = 1024;  // sequences per call supported by the score kernel
constexpr int kChunkBlocks = 64;
constexpr int kChunkBytes = kChunkBlocks * 2 * kHeadDim * 2;  // 32 KB
constexpr int kScoreSmem = kScoreStages * kChunkBytes + 1024 + 2 * kScoreStages * 8 + 64;

__global__ void __launch_bounds__(256, 1) score_kernel(CacheView c, const uint16_t* __restrict__ q,
                                                       float* __restrict__ scores) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t full0 = sbase + kScoreStages * kChunkBytes;
  const uint32_t empty0 = full0 + 8 * kScoreStages;
  // per-sequence block counts and the chunk prefix over (sequence, head) units
  __shared__ int sh_M[kMaxBatch];
  __shared__ int sh_pref[kMaxBatch + 1];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < kScoreStages; ++i) {
      mbar_init(full0 + 8 * i, 1);
      mbar_init(empty0 + 8 * i, kScoreWarps);
    }
    fence_mbar_init();
  }
  pdl_launch_dependents();
  pdl_wait();
  for (int b = tid; b < c.B; b += blockDim.x) {
    const int T = c.seq_lens[b];
    sh_M[b] = (T < 0 || T > c.max_blocks * kBlock) ? 0 : (T + kBlock - 1) / kBlock;  // bad lengths: top-n reports
  }
  __syncthreads();
  if (warp == 0) {  // exclusive prefix of Hkv * chunks-per-head over sequences
    int carry = 0;
    for (int b0 = 0; b0 < c.B; b0 += 32) {
      const int b = b0 + lane;
      const int v = b < c.B ? c.Hkv * ((sh_M[b] + kChunkBlocks - 1) / kChunkBlocks) : 0;
      int x = v;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
      }
      if (b < c.B) sh_pref[b] = carry + x - v;
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) sh_pref[c.B] = carry;
  }
  __syncthreads();
  const int total = sh_pref[c.B];
  const int per = (total + gridDim.x - 1) / gridDim.x;
  const int c0 = blockIdx.x * per, c1 = min(total, c0 + per);
  const int nmine = max(0, c1 - c0);

  // chunk index -> (sequence, head, first block, blocks): binary search of the prefix
  auto locate = [&](int ci, int& b, int& h, int& blk0, int& nblk) {
    int lo = 0, hi = c.B - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (sh_pref[mid] <= ci) lo = mid;
      else hi = mid - 1;
    }
    b = lo;
    const int M = sh_M[b];
    const int per_head = (M + kChunkBlocks - 1) / kChunkBlocks;
    const int r = ci - sh_pref[b];
    h = r / per_head;
    blk0 = (r % per_head) * kChunkBlocks;
    nblk = min(kChunkBlocks, M - blk0);
  };
  auto issue = [&](int k) {  // thread 0: my k-th chunk into stage k % kScoreStages
    int b, h, blk0, nblk;
    locate(c0 + k, b, h, blk0, nblk);
    const uint32_t bar = full0 + 8 * (k % kScoreStages);
    const uint32_t bytes = static_cast<uint32_t>(nblk) * 2 * kHeadDim * 2;
    mbar_arrive_expect_tx(bar, bytes);
    bulk_load(sbase + (k % kScoreStages) * kChunkBytes,
              c.summ + ((static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks + blk0) * 2 * kHeadDim, bytes, bar);
  };
  if (tid == 0)
    for (int k = 0; k < min(kScoreStages, nmine); ++k) issue(k);

  const int ch = lane & 15, half = lane >> 4;
  int cur_unit = -1;
  float qp[8];
  for (int k = 0; k < nmine; ++k) {
    const int st = k % kScoreStages;
    int b, h, blk0, nblk;
    locate(c0 + k, b, h, blk0, nblk);
    const int unit = b * c.Hkv + h;
    if (unit != cur_unit) {  // pooled query (mean of the group's heads), this lane's 8 dims
      cur_unit = unit;
#pragma unroll
      for (int j = 0; j < 8; ++j) qp[j] = 0.f;
      const uint16_t* qg = q + (static_cast<size_t>(b) * c.Hq + h * c.g) * kHeadDim + ch * 8;
      uint4 qv[kMaxGroup];  // all g rows in flight at once (g <= 8)
#pragma unroll
      for (int i = 0; i < kMaxGroup; ++i)
        qv[i] = i < c.g ? *reinterpret_cast<const uint4*>(qg + i * kHeadDim) : make_uint4(0, 0, 0, 0);
#pragma unroll
      for (int i = 0; i < kMaxGroup; ++i) {
        const uint32_t w[4] = {qv[i].x, qv[i].y, qv[i].z, qv[i].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          qp[2 * j] += bf16_lo(w[j]);
          qp[2 * j + 1] += bf16_hi(w[j]);
        }
      }
      const float inv_g = 1.0f / static_cast<float>(c.g);
#pragma unroll
      for (int j = 0; j < 8; ++j) qp[j] = qp[j] * inv_g;
    }
    int ok = 1;
    if (lane == 0) ok = mbar_wait_bounded(full0 + 8 * st, (k / kScoreStages) & 1) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (!ok) {
      if (lane == 0) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, unit);
      break;
    }
    mbar_try_wait(full0 + 8 * st, (k / kScoreStages) & 1);
    const uint8_t* chunk = smem + st * kChunkBytes;
    float* out = scores + static_cast<size_t>(unit) * c.max_blocks + blk0;
#pragma unroll
    for (int u = 0; u < kChunkBlocks / (2 * kScoreWarps); ++u) {
      const int blk = warp * (kChunkBlocks / kScoreWarps) + 2 * u + half;
      float sc = 0.f;
      if (blk < nblk) {
        const uint4 mn = *reinterpret_cast<const uint4*>(chunk + blk * 512 + ch * 16);
        const uint4 mx = *reinterpret_cast<const uint4*>(chunk + blk * 512 + 256 + ch * 16);
        sc = quest_term8(qp, mn, mx);
      }
      sc += __shfl_xor_sync(0xffffffffu, sc, 8);
      sc += __shfl_xor_sync(0xffffffffu, sc, 4);
      sc += __shfl_xor_sync(0xffffffffu, sc, 2);
      sc += __shfl_xor_sync(0xffffffffu, sc, 1);
      if (ch == 0 && blk < nblk) out[blk] = sc;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(empty0 + 8 * st);
    if (tid == 0 && k + kScoreStages < nmine) {
      // every warp has released this stage before it is refilled
      if (!mbar_wait_bounded(empty0 + 8 * st, (k / kScoreStages) & 1)) {
        record_error(c.status, RESA_DEV_WAIT_TIMEOUT, unit);
      } else {
        fence_proxy_async_smem();
        issue(k + kScoreStages);
      }
    }
  }
}

// Order-preserving map of an fp32 score to uint32 (larger score, larger key).
__device__ __forceinline__ uint32_t score_key(float s) {
  const uint32_t u = __float_as_uint(s);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive scan of one int per warp (kTopnWarps values, in place) by warp 0.
__device__ __forceinline__ void scan_warp_totals(int* vals) {
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < 32) {
    const int v = lane < kTopnWarps ? vals[lane] : 0;
    int x = v;
#pragma unroll
    for (int o = 1; o < kTopnWarps; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane < kTopnWarps) vals[lane] = x - v;
  }
}

// Cluster radix select, grid (kTopnCluster, KV head, sequence), one cluster
// per (sequence, KV head). CTA r stages the order-preserving keys of blocks
// [r * per, (r + 1) * per) in shared memory. Each 8-bit pass builds a local
// histogram of the keys that still match the prefix; after one cluster
// barrier every CTA sums the cluster's histograms through distributed shared
// memory and finds the same digit (histograms are double-buffered by pass
// parity, so one barrier per pass suffices). The select stops early when the
// boundary bucket is taken whole. Then each CTA counts its keys above the
// boundary and at it, reads the counts of the lower-ranked CTAs, and writes
// its selected ids in ascending order (ties at the boundary to the lower id).
__global__ void __launch_bounds__(kTopnThreads) topn_kernel(CacheView c, const float* __restrict__ scores,
                                                            double keep, int n_min, int n_local,
                                                            int32_t* __restrict__ indices,
                                                            int32_t* __restrict__ counts, int n_cap) {
  extern __shared__ uint32_t keys[];
  __shared__ int hist[2][256];
  __shared__ int tot[256];
  __shared__ int warp_a[kTopnWarps], warp_b[kTopnWarps];
  __shared__ int sh_digit, sh_rem, sh_done, sh_eq_before, sh_sel_before;
  __shared__ int cta_counts[2];  // keys above / at the boundary in this CTA, read by peers
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  pdl_launch_dependents();
  pdl_wait();
  const int rank = static_cast<int>(cluster.block_rank());
  const int b = blockIdx.z, h = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int32_t* out = indices + (static_cast<size_t>(b) * c.Hkv + h) * n_cap;
  const int T = c.seq_lens[b];
  if (T < 0 || T > c.max_blocks * kBlock) {  // the whole cluster takes this branch
    if (rank == 0 && tid == 0) {
      record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
      counts[b * c.Hkv + h] = 0;
    }
    for (int i = rank * kTopnThreads + tid; i < n_cap; i += kTopnCluster * kTopnThreads) out[i] = -1;
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
    if (rank == 0 && tid == 0) record_error(c.status, RESA_DEV_BUDGET_OVER_CAP, b * c.Hkv + h);
    n = n_cap;
  }
  const int per = (M + kTopnCluster - 1) / kTopnCluster;
  const int lo = rank * per, cnt = max(0, min(M, lo + per) - lo);
  const float* sc = scores + (static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks + lo;
  const int first_forced = M - n_local - lo;
  for (int i0 = 0; i0 < cnt; i0 += 4 * kTopnThreads) {  // four loads in flight per thread
    float v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u * kTopnThreads + tid;
      v[u] = i < cnt ? sc[i] : 0.f;
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = i0 + u * kTopnThreads + tid;
      if (i < cnt) keys[i] = (i >= first_forced) ? 0xFFFFFFFFu : score_key(v[u]);
    }
  }
  const int cnt_round = (cnt + 31) / 32 * 32;

  // ---- radix select of the n-th largest key across the cluster ----
  uint32_t prefix = 0, pmask = 0;
  int rem = n;
  __syncthreads();
  if (n > 0) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      int* hb = hist[pass & 1];
      hb[tid] = 0;
      __syncthreads();
      for (int i = tid; i < cnt_round; i += kTopnThreads) {
        uint32_t d = 0x100u;  // sentinel: not counted
        if (i < cnt) {
          const uint32_t k = keys[i];
          if ((k & pmask) == prefix) d = (k >> shift) & 0xFFu;
        }
        const unsigned peers = __match_any_sync(0xffffffffu, d);
        if (d != 0x100u && lane == __ffs(peers) - 1) atomicAdd(&hb[d], __popc(peers));
      }
      cluster.sync();  // every CTA's histogram of this pass is complete and visible
      int t = 0;
#pragma unroll
      for (int r = 0; r < kTopnCluster; ++r) t += cluster.map_shared_rank(hb, r)[tid];
      tot[tid] = t;
      __syncthreads();
      if (warp == 0) {
        // lane l owns digits 255-8l ... 248-8l (descending)
        int cn[8], sum = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          cn[j] = tot[255 - 8 * lane - j];
          sum += cn[j];
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
            if (cum + cn[j] >= rem) {
              sh_digit = 255 - 8 * lane - j;
              sh_rem = rem - cum;
              sh_done = (rem - cum == cn[j]) ? 1 : 0;  // the whole bucket is taken
              break;
            }
            cum += cn[j];
          }
        }
      }
      __syncthreads();
      prefix |= static_cast<uint32_t>(sh_digit) << shift;
      pmask |= 0xFFu << shift;
      rem = sh_rem;
      if (sh_done) break;  // identical decision in every CTA of the cluster
    }
  }
  // Selected: (key & pmask) > prefix, or == prefix among the first `take_eq`
  // such keys in block order.
  const int take_eq = n > 0 ? rem : 0;

  // ---- ordered compaction: warps own contiguous id ranges of the CTA ----
  const int per_warp = (cnt_round / 32 + kTopnWarps - 1) / kTopnWarps * 32;
  const int w0 = warp * per_warp, w1 = min(cnt, w0 + per_warp);
  int gt = 0, eq = 0;
  if (n > 0) {
    for (int i0 = w0; i0 < w0 + per_warp; i0 += 32) {
      const int i = i0 + lane;
      const bool in = i < w1;
      const uint32_t k = in ? (keys[i] & pmask) : 0u;
      gt += __popc(__ballot_sync(0xffffffffu, in && k > prefix));
      eq += __popc(__ballot_sync(0xffffffffu, in && k == prefix));
    }
  }
  if (lane == 0) {
    warp_a[warp] = eq;
    warp_b[warp] = gt;
  }
  __syncthreads();
  if (tid == 0) {
    int g2 = 0, e2 = 0;
    for (int w = 0; w < kTopnWarps; ++w) {
      g2 += warp_b[w];
      e2 += warp_a[w];
    }
    cta_counts[0] = g2;
    cta_counts[1] = e2;
  }
  cluster.sync();  // every CTA's counts are visible
  if (tid == 0) {
    int eq_before = 0, sel_before = 0;
    for (int r = 0; r < rank; ++r) {
      const int* pc = cluster.map_shared_rank(cta_counts, r);
      const int g2 = pc[0], e2 = pc[1];
      sel_before += g2 + max(0, min(e2, take_eq - eq_before));
      eq_before += e2;
    }
    sh_eq_before = eq_before;
    sh_sel_before = sel_before;
  }
  __syncthreads();
  scan_warp_totals(warp_a);  // exclusive prefix of equal keys per warp
  __syncthreads();
  if (lane == 0) {
    const int eq_b = sh_eq_before + warp_a[warp];
    warp_b[warp] = gt + max(0, min(eq, take_eq - eq_b));
  }
  __syncthreads();
  scan_warp_totals(warp_b);  // exclusive prefix of selected ids per warp
  __syncthreads();
  if (n > 0) {
    int eq_seen = sh_eq_before + warp_a[warp];
    int pos = sh_sel_before + warp_b[warp];
    for (int i0 = w0; i0 < w0 + per_warp; i0 += 32) {
      const int i = i0 + lane;
      const bool in = i < w1;
      const uint32_t k = in ? (keys[i] & pmask) : 0u;
      const bool is_eq = in && k == prefix;
      const unsigned eqm = __ballot_sync(0xffffffffu, is_eq);
      const int my_eq_rank = eq_seen + __popc(eqm & ((1u << lane) - 1u));
      const bool sel = in && (k > prefix || (is_eq && my_eq_rank < take_eq));
      const unsigned selm = __ballot_sync(0xffffffffu, sel);
      if (sel) out[pos + __popc(selm & ((1u << lane) - 1u))] = lo + i;
      eq_seen += __popc(eqm);
      pos += __popc(selm);
    }
  }
  for (int i = n + rank * kTopnThreads + tid; i < n_cap; i += kTopnCluster * kTopnThreads) out[i] = -1;
  if (rank == 0 && tid == 0) counts[b * c.Hkv + h] = n;
  cluster.sync();  // no CTA leaves while a peer may still read its counts
}

}  // namespace

size_t select_smem_bytes(int max_blocks) {
  return static_cast<size_t>((max_blocks + kTopnCluster - 1) / kTopnCluster) * sizeof(uint32_t);
}

int select_max_blocks() { return kTopnCluster * (kTopnSmemMax / static_cast<int>(sizeof(uint32_t))); }

cudaError_t launch_select(const CacheView& c, const uint16_t* q, double keep, int n_min, int n_local,
                          int32_t* indices, int32_t* counts, int n_cap, float* scores, int sm_count,
                          cudaStream_t st) {
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(score_kernel), kScoreSmem, 3);
  if (e != cudaSuccess) return e;
  // one persistent CTA per SM (never more than the chunks there can be)
  const int max_chunks = c.B * c.Hkv * ((c.max_blocks + kChunkBlocks - 1) / kChunkBlocks);
  const int grid = max(1, min(sm_count, max_chunks));
  e = launch_pdl(score_kernel, dim3(grid), dim3(kScoreWarps * 32), kScoreSmem, st, c, q, scores);
  if (e != cudaSuccess) return e;
  const size_t smem = select_smem_bytes(c.max_blocks);
  if (smem > 48 * 1024) {
    e = ensure_smem_attr(reinterpret_cast<const void*>(topn_kernel), kTopnSmemMax, 2);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kTopnCluster, c.Hkv, c.B);
  cfg.blockDim = dim3(kTopnThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = kTopnCluster;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, topn_kernel, c, static_cast<const float*>(scores), keep, n_min, n_local, indices,
                            counts, n_cap);
}

}  // namespace resa
