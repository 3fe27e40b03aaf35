// Block-sparse split-K flash decoding (Section 2.4; Algorithm 2) and the
// combine of split partials (Algorithm 2, "Combine").
//
// sparse_decode_kernel, grid (splits, KV head, sequence), 4 warps:
//   * The CTA owns index slots [s*per, (s+1)*per) of its (sequence, KV head),
//     per = ceil(n_cap / splits), and attends to the selected blocks among
//     them (slots below counts[b][h]). Warp w takes every 4th, so the group's
//     g <= 8 query heads share every K/V block fetched (GQA-shared fetch).
//   * Each warp streams its blocks through a private 3-stage shared-memory
//     ring: lane 0 issues four bulk-tensor TMA copies per block (K and V, two
//     64-column halves each, SWIZZLE_128B) that complete on the stage's
//     mbarrier. Swizzled rows make every ldmatrix below bank-conflict free.
//   * Per block (16 keys) the warp computes S^T = K * Q^T with 8
//     m16n8k16 bf16 MMAs (M = 16 keys, N = 8 heads, K = 128 dims), masks keys
//     at positions >= T, runs the online softmax in the log2 domain, moves
//     P^T from the accumulator layout to the B-operand layout with movmatrix,
//     and accumulates O^T += V^T * P^T with 8 more MMAs (V^T via ldmatrix.trans).
//   * The 4 warps' (m, l, O) are merged through shared memory; the CTA writes
//     a normalised partial O (fp32) and its log2-sum-exp for each head.
// merge_kernel, one CTA per output row: LSE-weighted sum of the split partials
// (merge_rows_kernel, one warp per row, for calls of many rows and few splits).
#include <atomic>

#include "resa_device.cuh"
#include "resa_launch.h"

namespace resa {
namespace {

constexpr int kWarps = 4;
constexpr int kStages = 3;
constexpr int kStageBytes = 8192;  // K: 2 x 2 KB halves, V: 2 x 2 KB halves
constexpr int kRingBytes = kWarps * kStages * kStageBytes;
constexpr int kDecodeSmem = kRingBytes + 1024 /* alignment slack */ + kWarps * kStages * 8;
constexpr float kNegInf = -__builtin_huge_valf();
constexpr float kLazyLog2 = 8.f;  // base moves when a score exceeds it by more than 2^8

struct DecodeArgs {
  const uint16_t* q;
  const int32_t* indices;
  const int32_t* counts;
  int n_cap;
  int splits;
  float scale_log2;
  float* o_part;    // [B][Hq][splits][128]
  float* lse_part;  // [B][Hq][splits], log2 domain
  uint32_t wait_polls;  // polls of a copy's barrier before the warp gives up (the drain keeps kWaitPolls)
};

__device__ __forceinline__ float safe_base(float m) { return m == kNegInf ? 0.f : m; }

__global__ void __launch_bounds__(kWarps * 32) sparse_decode_kernel(const __grid_constant__ CUtensorMap tm_k,
                                                                    const __grid_constant__ CUtensorMap tm_v,
                                                                    CacheView c, DecodeArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kRingBytes);
  __shared__ float wm[kWarps][8], wl[kWarps][8];

  const int s = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t ring = smem_u32(smem) + warp * kStages * kStageBytes;
  const uint32_t bar0 = smem_u32(bars + warp * kStages);
  if (lane == 0) {
    for (int st = 0; st < kStages; ++st) mbar_init(bar0 + 8 * st, 1);
    fence_mbar_init();
    prefetch_tmap(&tm_k);
    prefetch_tmap(&tm_v);
  }
  __syncwarp();
  pdl_launch_dependents();
  pdl_wait();
  // Splits cover the index capacity [0, n_cap): the CTA's id range is known
  // before `counts` arrives, so ids, length, count and queries load together.
  const int per = (a.n_cap + a.splits - 1) / a.splits;
  const int j0 = s * per;
  const int nj_cap = max(0, min(a.n_cap, j0 + per) - j0);
  const int cnt_cap = nj_cap > warp ? (nj_cap - warp + kWarps - 1) / kWarps : 0;
  const int32_t* idx = a.indices + static_cast<size_t>(b * c.Hkv + h) * a.n_cap + j0 + warp;
  const int T = c.seq_lens[b] + c.pending;
  int n = a.counts[b * c.Hkv + h];
  int pre_blk = lane < cnt_cap ? idx[lane * kWarps] : -1;
  if (T < 0 || T > c.max_blocks * kBlock) {
    if (threadIdx.x == 0 && s == 0) record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
    n = 0;
  } else if (n < 0 || n > a.n_cap) {
    if (threadIdx.x == 0 && s == 0) record_error(c.status, RESA_DEV_BAD_INDEX, b * c.Hkv + h);
    n = 0;
  }
  const int M = (max(T, 0) + kBlock - 1) / kBlock;
  // this warp's blocks are ids j0 + warp + kWarps * it < n
  const int cnt = max(0, min(cnt_cap, (n - j0 - warp + kWarps - 1) / kWarps));

  // Page of block blk, or -1 if the id is out of range, -2 if its page is.
  // Such blocks are fully masked (and reported).
  auto page_of = [&](int blk) -> int {
    if (blk < 0 || blk >= M) return -1;
    const int page = c.page_table[static_cast<size_t>(b) * c.max_blocks + blk];
    return (page >= 0 && page < c.num_pages) ? page : -2;
  };
  int pre_page = -1;
  if (lane < cnt) pre_page = page_of(pre_blk);
  auto info = [&](int it, int& blk) -> int {  // warp-uniform; ids beyond 32 per warp load on demand
    if (it < 32) {
      blk = __shfl_sync(0xffffffffu, pre_blk, it);
      return __shfl_sync(0xffffffffu, pre_page, it);
    }
    blk = idx[it * kWarps];
    return page_of(blk);
  };
  auto issue = [&](int it, int st) {  // warp-uniform; lane 0 issues
    int blk;
    const int page = info(it, blk);
    if (lane != 0) return;
    const uint32_t bar = bar0 + 8 * st;
    if (page < 0) {
      record_error(c.status, page == -1 ? RESA_DEV_BAD_INDEX : RESA_DEV_PAGE_RANGE, b * c.Hkv + h);
      mbar_arrive(bar);  // completes the phase with no data
      return;
    }
    const int row = (page * c.Hkv + h) * kBlock;
    const uint32_t dst = ring + st * kStageBytes;
    mbar_arrive_expect_tx(bar, kStageBytes);
    tma_load_2d_stream(dst, &tm_k, bar, 0, row);
    tma_load_2d_stream(dst + 2048, &tm_k, bar, 64, row);
    tma_load_2d_stream(dst + 4096, &tm_v, bar, 0, row);
    tma_load_2d_stream(dst + 6144, &tm_v, bar, 64, row);
  };

  // Q^T as the B operand: lane holds head lane/4, dims 16ks + 2(lane%4) (+1, +8, +9).
  uint32_t qb[8][2];
  {
    const int qh = lane >> 2;
    const bool ok = qh < c.g;
    const uint16_t* qr = a.q + (static_cast<size_t>(b) * c.Hq + h * c.g + (ok ? qh : 0)) * kHeadDim;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      const int d0 = 16 * ks + 2 * (lane & 3);
      qb[ks][0] = ok ? *reinterpret_cast<const uint32_t*>(qr + d0) : 0u;
      qb[ks][1] = ok ? *reinterpret_cast<const uint32_t*>(qr + d0 + 8) : 0u;
    }
  }

  int issued = 0;
  for (; issued < min(kStages, cnt); ++issued) issue(issued, issued);

  float m0 = kNegInf, m1 = kNegInf, l0 = 0.f, l1 = 0.f;
  float acc[8][4];
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) acc[mt][0] = acc[mt][1] = acc[mt][2] = acc[mt][3] = 0.f;

  int it = 0;
  for (; it < cnt; ++it) {
    const int st = it % kStages;
    const uint32_t par = (it / kStages) & 1;
    const uint32_t bar = bar0 + 8 * st;
    int ok = 1;
    if (lane == 0) ok = mbar_wait_polls(bar, par, a.wait_polls) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (!ok) {
      if (lane == 0) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, b * c.Hkv + h);
      break;
    }
    mbar_try_wait(bar, par);  // acquire for every lane (the phase has completed)
    int blk;
    const int page = info(it, blk);
    const int valid = page < 0 ? 0 : min(kBlock, T - blk * kBlock);
    const uint32_t kb = ring + st * kStageBytes, vb = kb + 4096;
    if (valid < kBlock) {  // rows past the end (or an invalid block) may hold garbage: zero V
      uint8_t* v = smem + (kb - smem_u32(smem)) + 4096;
      for (int e = lane; e < (kBlock - valid) * 16; e += 32) {
        const int r = valid + (e >> 4), half = (e >> 3) & 1, chunk = e & 7;
        *reinterpret_cast<uint4*>(v + half * 2048 + r * 128 + chunk * 16) = make_uint4(0, 0, 0, 0);
      }
      __syncwarp();
    }
    // S^T = K * Q^T
    float sc[4] = {0.f, 0.f, 0.f, 0.f};
    {
      // two accumulators (even / odd k-steps) halve the dependent MMA chain
      float sd[4] = {0.f, 0.f, 0.f, 0.f};
      const int key = (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int chunk = 2 * ks + (lane >> 4);
        uint32_t a0, a1, a2, a3;
        ldsm_x4(kb + (chunk >> 3) * 2048 + sw128(key, chunk & 7), a0, a1, a2, a3);
        mma_bf16_16816((ks & 1) ? sd : sc, a0, a1, a2, a3, qb[ks][0], qb[ks][1]);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) sc[i] += sd[i];
    }
    const int k0 = lane >> 2;
    float s0 = (k0 < valid) ? sc[0] * a.scale_log2 : kNegInf;
    float s1 = (k0 < valid) ? sc[1] * a.scale_log2 : kNegInf;
    float s2 = (k0 + 8 < valid) ? sc[2] * a.scale_log2 : kNegInf;
    float s3 = (k0 + 8 < valid) ? sc[3] * a.scale_log2 : kNegInf;
    // Lazy base: a head's base (m) moves only when one of the block's scores
    // exceeds it by more than 2^8 (then to the exact running maximum, with O
    // and l rescaled); otherwise the block needs no cross-lane maximum and no
    // rescale. P = 2^(s - m) <= 2^8 is exact in range for bf16 and fp32.
    if (__any_sync(0xffffffffu, s0 > m0 + kLazyLog2 || s2 > m0 + kLazyLog2 || s1 > m1 + kLazyLog2 ||
                                    s3 > m1 + kLazyLog2)) {
      float bm0 = fmaxf(s0, s2), bm1 = fmaxf(s1, s3);
#pragma unroll
      for (int o = 4; o < 32; o <<= 1) {
        bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, o));
        bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, o));
      }
      const float n0 = fmaxf(m0, bm0), n1 = fmaxf(m1, bm1);
      const float al0 = exp2f(m0 - safe_base(n0)), al1 = exp2f(m1 - safe_base(n1));
      l0 *= al0;
      l1 *= al1;
      m0 = n0;
      m1 = n1;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        acc[mt][0] *= al0;
        acc[mt][1] *= al1;
        acc[mt][2] *= al0;
        acc[mt][3] *= al1;
      }
    }
    const float base0 = safe_base(m0), base1 = safe_base(m1);
    const uint32_t x0 = pack_bf16x2(exp2f(s0 - base0), exp2f(s1 - base1));
    const uint32_t x1 = pack_bf16x2(exp2f(s2 - base0), exp2f(s3 - base1));
    l0 += bf16_lo(x0) + bf16_lo(x1);
    l1 += bf16_hi(x0) + bf16_hi(x1);
    const uint32_t pb0 = movmatrix_t(x0), pb1 = movmatrix_t(x1);
    // O^T += V^T * P^T
    {
      const int j = lane >> 3;
      const int key = (lane & 7) + (j >> 1) * 8;
#pragma unroll
      for (int mt = 0; mt < 8; ++mt) {
        const int chunk = 2 * mt + (j & 1);
        uint32_t a0, a1, a2, a3;
        ldsm_x4_t(vb + (chunk >> 3) * 2048 + sw128(key, chunk & 7), a0, a1, a2, a3);
        mma_bf16_16816(acc[mt], a0, a1, a2, a3, pb0, pb1);
      }
    }
    __syncwarp();
    if (issued < cnt) {
      if (lane == 0) fence_proxy_async_smem();
      issue(issued, st);
      ++issued;
    }
  }
  if (it < cnt && lane == 0) {  // timed out: let copies already in flight land (default limit) before leaving
    for (int k = it; k < issued; ++k) mbar_wait_bounded(bar0 + 8 * (k % kStages), (k / kStages) & 1);
  }

  // ---- merge the 4 warps' softmax states ----
#pragma unroll
  for (int o = 4; o < 32; o <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, o);
    l1 += __shfl_xor_sync(0xffffffffu, l1, o);
  }
  if (lane < 4) {
    wm[warp][2 * lane] = m0;
    wm[warp][2 * lane + 1] = m1;
    wl[warp][2 * lane] = l0;
    wl[warp][2 * lane + 1] = l1;
  }
  __syncthreads();
  const int hA = 2 * (lane & 3), hB = hA + 1;
  float MA = kNegInf, MB = kNegInf;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    MA = fmaxf(MA, wm[w][hA]);
    MB = fmaxf(MB, wm[w][hB]);
  }
  float LA = 0.f, LB = 0.f;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    LA += wl[w][hA] * exp2f(wm[w][hA] - safe_base(MA));
    LB += wl[w][hB] * exp2f(wm[w][hB] - safe_base(MB));
  }
  const float fA = LA > 0.f ? exp2f(m0 - safe_base(MA)) / LA : 0.f;
  const float fB = LB > 0.f ? exp2f(m1 - safe_base(MB)) / LB : 0.f;
  constexpr int kRedRow = kHeadDim + 4;  // padded: the four heads a warp writes at once fall in distinct banks
  float* red = reinterpret_cast<float*>(smem);  // [warp][8 heads][kRedRow] fp32, reuses the ring
#pragma unroll
  for (int mt = 0; mt < 8; ++mt) {
    const int dA = 16 * mt + (lane >> 2), dB = dA + 8;
    red[(warp * 8 + hA) * kRedRow + dA] = acc[mt][0] * fA;
    red[(warp * 8 + hB) * kRedRow + dA] = acc[mt][1] * fB;
    red[(warp * 8 + hA) * kRedRow + dB] = acc[mt][2] * fA;
    red[(warp * 8 + hB) * kRedRow + dB] = acc[mt][3] * fB;
  }
  __syncthreads();
  const int t = threadIdx.x;
  for (int hh = 0; hh < c.g; ++hh) {
    const size_t row = static_cast<size_t>(b) * c.Hq + h * c.g + hh;
    for (int dd = t; dd < kHeadDim; dd += kWarps * 32) {  // output dims of this thread
      float v = 0.f;
#pragma unroll
      for (int w = 0; w < kWarps; ++w) v += red[(w * 8 + hh) * kRedRow + dd];
      a.o_part[(row * a.splits + s) * kHeadDim + dd] = v;
    }
  }
  if (t < c.g) {
    float Mt = kNegInf;
    for (int w = 0; w < kWarps; ++w) Mt = fmaxf(Mt, wm[w][t]);
    float Lt = 0.f;
    for (int w = 0; w < kWarps; ++w) Lt += wl[w][t] * exp2f(wm[w][t] - safe_base(Mt));
    const size_t row = static_cast<size_t>(b) * c.Hq + h * c.g + t;
    a.lse_part[row * a.splits + s] = Lt > 0.f ? Mt + log2f(Lt) : kNegInf;
  }
}

// Length advance of a fused decode step: the merge is its last kernel, so it
// counts the appended token in seq_lens (row 0 of each sequence; a length
// that the call found out of range is left as it is).
struct LenAdvance {
  int32_t* lens;  // null: no advance
  int pending;
  int cap;        // max_blocks * 16
};

// One CTA of 8 warps per output row. Warp w takes the splits w, w + 8, ...:
// its lanes load ten partial rows (16 bytes each) and their log2-sum-exps at
// once, so up to 80 splits cost one round of loads; each warp keeps its sum
// relative to its own maximum, and the warps' maxima and rows are combined
// through shared memory.
constexpr int kMergeWarps = 8;
constexpr int kRowMergeMinRows = 1024;  // calls with at least this many rows (and <= 16 splits) merge a row per warp

// kLoads partial rows in flight per lane (8 kLoads splits in one round); the
// launch picks the smallest instantiation of at least 4 that covers the
// splits in one round (up to 80; more take further rounds with an online
// rescale). The 1- and 2-load forms measured slower in the fused decode
// step although they do less work; with fewer registers, more of the merge
// CTAs launched early can be placed on each SM beside the decode CTAs, so
// the merge would run on fewer SMs (the likely cause).
template <int kLoads>
__global__ void __launch_bounds__(kMergeWarps * 32) merge_kernel(const float* __restrict__ o_part,
                                                                 const float* __restrict__ lse_part, int splits,
                                                                 uint16_t* __restrict__ out,
                                                                 float* __restrict__ lse_out,
                                                                 const int32_t* __restrict__ active,
                                                                 int rows_per_seq, LenAdvance adv) {
  __shared__ float4 red[kMergeWarps][kHeadDim / 4];
  __shared__ float wmax[kMergeWarps], wsum[kMergeWarps];
  pdl_launch_dependents();
  pdl_wait();
  const size_t row = blockIdx.x;
  if (adv.lens != nullptr && threadIdx.x == 0 && row % rows_per_seq == 0) {
    const int b = static_cast<int>(row / rows_per_seq);
    const int T = adv.lens[b];
    if (T >= 0 && T + adv.pending <= adv.cap) adv.lens[b] = T + adv.pending;
  }
  if (active != nullptr && active[row / rows_per_seq] == 0) return;  // a sequence left out of the call
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float* lp = lse_part + row * splits;
  const float4* op = reinterpret_cast<const float4*>(o_part + row * splits * kHeadDim) + lane;
  // this warp's splits w + 8 j and their log2-sum-exps, kLoads of each in
  // flight together; the warp's weighted sum of rows (acc) and of weights
  // (l, the normaliser's share) are relative to its running maximum m
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float m = kNegInf, l = 0.f;
  for (int base = 0; base < splits; base += kMergeWarps * kLoads) {
    float4 v[kLoads];
    float ls[kLoads];
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {
      const int sp = base + warp + kMergeWarps * j;
      const bool ok = sp < splits;
      v[j] = ok ? op[static_cast<size_t>(sp) * (kHeadDim / 4)] : make_float4(0.f, 0.f, 0.f, 0.f);
      ls[j] = ok ? lp[sp] : kNegInf;
    }
    float mb = m;
#pragma unroll
    for (int j = 0; j < kLoads; ++j) mb = fmaxf(mb, ls[j]);
    const float sc = m == kNegInf ? 0.f : exp2f(m - safe_base(mb));
    acc.x *= sc;
    acc.y *= sc;
    acc.z *= sc;
    acc.w *= sc;
    l *= sc;
    m = mb;
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {
      const float w = exp2f(ls[j] - safe_base(m));
      acc.x += w * v[j].x;
      acc.y += w * v[j].y;
      acc.z += w * v[j].z;
      acc.w += w * v[j].w;
      l += w;
    }
  }
  // acc is this warp's sum relative to its own maximum m: rescale to the CTA's
  if (lane == 0) wmax[warp] = m;
  __syncthreads();
  float M = kNegInf;
#pragma unroll
  for (int w = 0; w < kMergeWarps; ++w) M = fmaxf(M, wmax[w]);
  const float sc = m == kNegInf ? 0.f : exp2f(m - safe_base(M));
  acc.x *= sc; acc.y *= sc; acc.z *= sc; acc.w *= sc;
  red[warp][lane] = acc;
  if (lane == 0) wsum[warp] = l * sc;
  __syncthreads();
  if (warp == 0) {
    float4 t = red[0][lane];
#pragma unroll
    for (int w = 1; w < kMergeWarps; ++w) {
      t.x += red[w][lane].x;
      t.y += red[w][lane].y;
      t.z += red[w][lane].z;
      t.w += red[w][lane].w;
    }
    // the normaliser: the warps' weight sums, relative to M
    float l = 0.f;
#pragma unroll
    for (int w = 0; w < kMergeWarps; ++w) l += wsum[w];
    const float inv = l > 0.f ? 1.f / l : 0.f;
    uint2 packed;
    packed.x = pack_bf16x2(t.x * inv, t.y * inv);
    packed.y = pack_bf16x2(t.z * inv, t.w * inv);
    *reinterpret_cast<uint2*>(out + row * kHeadDim + 4 * lane) = packed;
    if (lse_out != nullptr && lane == 0) lse_out[row] = l > 0.f ? (M + log2f(l)) * 0.69314718055994530942f : kNegInf;
  }
}

// One warp per output row, for calls with many rows and few splits (the
// rectification's partials: B f Hq rows of a few splits each), where a CTA
// per row would leave most of its warps idle: lane l holds dims 4l .. 4l + 3
// of kLoads partial rows in flight and the warp keeps the running maximum,
// the weighted row sum and the weight sum (an online rescale between rounds
// when there are more than kLoads splits). No shared memory, no barrier.
template <int kLoads>
__global__ void __launch_bounds__(kMergeWarps * 32) merge_rows_kernel(const float* __restrict__ o_part,
                                                                      const float* __restrict__ lse_part,
                                                                      int splits, int rows, uint16_t* __restrict__ out,
                                                                      float* __restrict__ lse_out,
                                                                      const int32_t* __restrict__ active,
                                                                      int rows_per_seq, LenAdvance adv) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const size_t row = static_cast<size_t>(blockIdx.x) * kMergeWarps + (threadIdx.x >> 5);
  if (row >= static_cast<size_t>(rows)) return;
  if (adv.lens != nullptr && lane == 0 && row % rows_per_seq == 0) {
    const int b = static_cast<int>(row / rows_per_seq);
    const int T = adv.lens[b];
    if (T >= 0 && T + adv.pending <= adv.cap) adv.lens[b] = T + adv.pending;
  }
  if (active != nullptr && active[row / rows_per_seq] == 0) return;  // a sequence left out of the call
  const float* lp = lse_part + row * splits;
  const float4* op = reinterpret_cast<const float4*>(o_part + row * splits * kHeadDim) + lane;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float m = kNegInf, l = 0.f;
  for (int base = 0; base < splits; base += kLoads) {
    float4 v[kLoads];
    float ls[kLoads];
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {
      const int sp = base + j;
      const bool ok = sp < splits;
      v[j] = ok ? op[static_cast<size_t>(sp) * (kHeadDim / 4)] : make_float4(0.f, 0.f, 0.f, 0.f);
      ls[j] = ok ? lp[sp] : kNegInf;
    }
    float mb = m;
#pragma unroll
    for (int j = 0; j < kLoads; ++j) mb = fmaxf(mb, ls[j]);
    const float sc = m == kNegInf ? 0.f : exp2f(m - safe_base(mb));
    acc.x *= sc;
    acc.y *= sc;
    acc.z *= sc;
    acc.w *= sc;
    l *= sc;
    m = mb;
#pragma unroll
    for (int j = 0; j < kLoads; ++j) {
      const float w = exp2f(ls[j] - safe_base(m));
      acc.x += w * v[j].x;
      acc.y += w * v[j].y;
      acc.z += w * v[j].z;
      acc.w += w * v[j].w;
      l += w;
    }
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
  uint2 packed;
  packed.x = pack_bf16x2(acc.x * inv, acc.y * inv);
  packed.y = pack_bf16x2(acc.z * inv, acc.w * inv);
  *reinterpret_cast<uint2*>(out + row * kHeadDim + 4 * lane) = packed;
  if (lse_out != nullptr && lane == 0) lse_out[row] = l > 0.f ? (m + log2f(l)) * 0.69314718055994530942f : kNegInf;
}

}  // namespace

int decode_ctas_per_sm() {
  static std::atomic<int> cached{0};
  int v = cached.load(std::memory_order_relaxed);
  if (v > 0) return v;
  if (ensure_smem_attr(reinterpret_cast<const void*>(sparse_decode_kernel), kDecodeSmem, 0) != cudaSuccess) return 1;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, sparse_decode_kernel, kWarps * 32, kDecodeSmem) !=
          cudaSuccess ||
      n < 1)
    n = 1;
  cached.store(n, std::memory_order_relaxed);
  return n;
}

cudaError_t launch_sparse_decode(const CacheView& c, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                                 const uint16_t* q, const int32_t* indices, const int32_t* counts, int n_cap,
                                 float sm_scale, int splits, float* o_part, float* lse_part, cudaStream_t st,
                                 uint32_t wait_polls) {
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(sparse_decode_kernel), kDecodeSmem, 0);
  if (e != cudaSuccess) return e;
  DecodeArgs a{q,        indices,  counts, n_cap, splits, sm_scale * 1.44269504088896340736f,
               o_part,   lse_part, wait_polls};
  return launch_pdl(sparse_decode_kernel, dim3(splits, c.Hkv, c.B), dim3(kWarps * 32), kDecodeSmem, st, tm_k,
                    tm_v, c, a);
}

cudaError_t launch_merge(const float* o_part, const float* lse_part, int rows, int splits, uint16_t* out,
                         float* lse_out, cudaStream_t st, const int32_t* active, int rows_per_seq,
                         const CacheView* advance) {
  if (rows == 0) return cudaSuccess;
  LenAdvance adv{nullptr, 0, 0};
  if (advance != nullptr && advance->pending > 0)
    adv = LenAdvance{advance->seq_lens, advance->pending, advance->max_blocks * kBlock};
  if (rows >= kRowMergeMinRows && splits <= 16) {
    // many rows of few splits: a warp per row, all of a row's splits in flight
    const auto kernel = splits <= 4 ? merge_rows_kernel<4> : splits <= 8 ? merge_rows_kernel<8> : merge_rows_kernel<16>;
    return launch_pdl(kernel, dim3((rows + kMergeWarps - 1) / kMergeWarps), dim3(kMergeWarps * 32), 0, st, o_part,
                      lse_part, splits, rows, out, lse_out, active, rows_per_seq, adv);
  }
  const int per_warp = (splits + kMergeWarps - 1) / kMergeWarps;
  const auto kernel = per_warp <= 4 ? merge_kernel<4>
                      : per_warp <= 6 ? merge_kernel<6>
                                      : merge_kernel<10>;
  return launch_pdl(kernel, dim3(rows), dim3(kMergeWarps * 32), 0, st, o_part, lse_part, splits, out, lse_out,
                    active, rows_per_seq, adv);
}

}  // namespace resa
