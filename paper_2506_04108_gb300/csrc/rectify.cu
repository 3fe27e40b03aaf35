// Dense rectification attention (Section 2.2; Algorithm 1 DenseForward).
//
// For each (sequence b, KV head h) the g*f query rows of the group (row
// r = i*g + j: token i of the f, query head h*g + j, position T - f + i)
// attend causally to the whole cache. Work split:
//   grid (key splits, row groups of 128, sequence * KV head), 8 warps,
//   warp w owns 16 query rows; the CTA streams 64-key tiles of the prefix
//   [0, T - f) from the paged cache with bulk-tensor TMA (SWIZZLE_128B,
//   one copy per 16-key page per 64-column half) into a 2-stage ring, and
//   the last split also takes the f-token tail from k_new / v_new with the
//   causal mask (key t of the tail is visible to token i iff t <= i).
//   S = Q K^T and O += P V run on m16n8k16 bf16 MMAs with fp32 accumulation
//   and an online softmax in the log2 domain; each split writes a
//   normalised partial O and its log2-sum-exp, combined by merge_kernel.
#include "resa_device.cuh"
#include "resa_launch.h"

namespace resa {
namespace {

constexpr int kWarps = 8;
constexpr int kRows = 16 * kWarps;  // query rows per CTA
constexpr int kTile = 64;           // keys per tile
constexpr int kHalfBytes = kTile * 128;       // one 64-column half of a tile
constexpr int kStageBytes = 4 * kHalfBytes;   // K (2 halves) + V (2 halves) = 32 KB
constexpr int kStages = 2;
constexpr int kSmem = kStages * kStageBytes + 1024 + 64;
constexpr float kNegInf = -__builtin_huge_valf();

struct RectArgs {
  const uint16_t* q_new;  // [B][f][Hq][128]
  const uint16_t* k_new;  // [B][f][Hkv][128]
  const uint16_t* v_new;
  int f;
  int splits;
  float scale_log2;
  float* o_part;    // [B*f*Hq][splits][128]
  float* lse_part;  // [B*f*Hq][splits], log2 domain
};

__device__ __forceinline__ float safe_base(float m) { return m == kNegInf ? 0.f : m; }

__global__ void __launch_bounds__(kWarps * 32, 1) rectify_kernel(const __grid_constant__ CUtensorMap tm_k,
                                                                 const __grid_constant__ CUtensorMap tm_v,
                                                                 CacheView c, RectArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  __shared__ int sh_ok;

  const int s = blockIdx.x, rg = blockIdx.y, bh = blockIdx.z;
  const int b = bh / c.Hkv, h = bh % c.Hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int f = a.f, g = c.g;
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = smem_u32(bars);
  if (tid == 0) {
    for (int st = 0; st < kStages; ++st) mbar_init(bar0 + 8 * st, 1);
    fence_mbar_init();
    prefetch_tmap(&tm_k);
    prefetch_tmap(&tm_v);
  }
  __syncthreads();
  pdl_launch_dependents();
  pdl_wait();
  const int T = c.seq_lens[b];
  if (T < f || T > c.max_blocks * kBlock) {
    if (tid == 0 && s == 0 && rg == 0) record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
    return;
  }
  const int P = T - f;                         // prefix keys from the cache
  const int ntp = (P + kTile - 1) / kTile;     // prefix tiles
  const int per = (ntp + a.splits - 1) / a.splits;
  const int t0 = s * per;
  const int n_pref = max(0, min(ntp, t0 + per) - t0);
  const int n_tail = (s == a.splits - 1) ? (f + kTile - 1) / kTile : 0;
  const int R = g * f;

  auto issue = [&](int lt, int st) {  // thread 0: prefix tile t0 + lt into stage st
    const int kb = (t0 + lt) * kTile;
    const uint32_t bar = bar0 + 8 * st;
    const uint32_t dk = sbase + st * kStageBytes, dv = dk + 2 * kHalfBytes;
    int pages = 0, rows[4];
    for (int pg = 0; pg < 4; ++pg) {
      rows[pg] = -1;
      const int blk = kb / kBlock + pg;
      if (blk * kBlock >= P) continue;
      const int page = c.page_table[static_cast<size_t>(b) * c.max_blocks + blk];
      if (page < 0 || page >= c.num_pages) {
        record_error(c.status, RESA_DEV_PAGE_RANGE, b);
        continue;
      }
      rows[pg] = (page * c.Hkv + h) * kBlock;
      ++pages;
    }
    mbar_arrive_expect_tx(bar, pages * 4 * 2048);
    for (int pg = 0; pg < 4; ++pg) {
      if (rows[pg] < 0) continue;
      const uint32_t o = pg * 2048;
      tma_load_2d(dk + o, &tm_k, bar, 0, rows[pg]);
      tma_load_2d(dk + kHalfBytes + o, &tm_k, bar, 64, rows[pg]);
      tma_load_2d(dv + o, &tm_v, bar, 0, rows[pg]);
      tma_load_2d(dv + kHalfBytes + o, &tm_v, bar, 64, rows[pg]);
    }
  };
  if (tid == 0)
    for (int lt = 0; lt < min(kStages, n_pref); ++lt) issue(lt, lt);

  // Q rows of this thread: rA = row0 + 16*warp + lane/4, rB = rA + 8.
  const int rA = rg * kRows + warp * 16 + (lane >> 2), rB = rA + 8;
  const int iA = rA < R ? rA / g : -1, iB = rB < R ? rB / g : -1;
  uint32_t qa[8][4];
  {
    const uint16_t* qA = a.q_new + ((static_cast<size_t>(b) * f + max(iA, 0)) * c.Hq + h * g + rA % g) * kHeadDim;
    const uint16_t* qB = a.q_new + ((static_cast<size_t>(b) * f + max(iB, 0)) * c.Hq + h * g + rB % g) * kHeadDim;
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
      const int d0 = 16 * ks + 2 * (lane & 3);
      qa[ks][0] = iA >= 0 ? *reinterpret_cast<const uint32_t*>(qA + d0) : 0u;
      qa[ks][1] = iB >= 0 ? *reinterpret_cast<const uint32_t*>(qB + d0) : 0u;
      qa[ks][2] = iA >= 0 ? *reinterpret_cast<const uint32_t*>(qA + d0 + 8) : 0u;
      qa[ks][3] = iB >= 0 ? *reinterpret_cast<const uint32_t*>(qB + d0 + 8) : 0u;
    }
  }

  float mA = kNegInf, mB = kNegInf, lA = 0.f, lB = 0.f;
  float o[16][4];
#pragma unroll
  for (int nt = 0; nt < 16; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;

  // One 64-key tile held in stage `st`. Key column c is visible to row r iff
  // visible(c, i(r)): prefix tiles: kb + c < P; tail tiles: tb + c < f && tb + c <= i.
  auto tile = [&](int st, bool tail, int kbase) {
    const uint32_t kst = sbase + st * kStageBytes, vst = kst + 2 * kHalfBytes;
    float sc[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
    {
      const int j = lane >> 3, r = lane & 7;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        const int chunk = 2 * ks + (j & 1);
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          const int key = 16 * np + r + 8 * (j >> 1);
          uint32_t b0, b1, b2, b3;
          ldsm_x4(kst + (chunk >> 3) * kHalfBytes + sw128(key, chunk & 7), b0, b1, b2, b3);
          mma_bf16_16816(sc[2 * np], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], b0, b1);
          mma_bf16_16816(sc[2 * np + 1], qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3], b2, b3);
        }
      }
    }
    float tmA = kNegInf, tmB = kNegInf;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int col = kbase + 8 * nt + 2 * (lane & 3) + e;
        const bool vA = tail ? (col < f && col <= iA) : (col < P);
        const bool vB = tail ? (col < f && col <= iB) : (col < P);
        sc[nt][e] = vA ? sc[nt][e] * a.scale_log2 : kNegInf;
        sc[nt][2 + e] = vB ? sc[nt][2 + e] * a.scale_log2 : kNegInf;
        tmA = fmaxf(tmA, sc[nt][e]);
        tmB = fmaxf(tmB, sc[nt][2 + e]);
      }
    }
#pragma unroll
    for (int x = 1; x < 4; x <<= 1) {
      tmA = fmaxf(tmA, __shfl_xor_sync(0xffffffffu, tmA, x));
      tmB = fmaxf(tmB, __shfl_xor_sync(0xffffffffu, tmB, x));
    }
    const float nA = fmaxf(mA, tmA), nB = fmaxf(mB, tmB);
    const float baseA = safe_base(nA), baseB = safe_base(nB);
    const float alA = exp2f(mA - baseA), alB = exp2f(mB - baseB);
    mA = nA;
    mB = nB;
    uint32_t pa[4][4];
    float sumA = 0.f, sumB = 0.f;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        const int nt = 2 * kk + hf;
        const uint32_t xa = pack_bf16x2(exp2f(sc[nt][0] - baseA), exp2f(sc[nt][1] - baseA));
        const uint32_t xb = pack_bf16x2(exp2f(sc[nt][2] - baseB), exp2f(sc[nt][3] - baseB));
        sumA += bf16_lo(xa) + bf16_hi(xa);
        sumB += bf16_lo(xb) + bf16_hi(xb);
        pa[kk][2 * hf] = xa;
        pa[kk][2 * hf + 1] = xb;
      }
    }
    lA = lA * alA + sumA;
    lB = lB * alB + sumB;
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) {
      o[nt][0] *= alA;
      o[nt][1] *= alA;
      o[nt][2] *= alB;
      o[nt][3] *= alB;
    }
    {
      const int j = lane >> 3, r = lane & 7;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        const int key = 16 * kk + r + 8 * (j & 1);
#pragma unroll
        for (int dp = 0; dp < 8; ++dp) {
          const int chunk = 2 * dp + (j >> 1);
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(vst + (chunk >> 3) * kHalfBytes + sw128(key, chunk & 7), b0, b1, b2, b3);
          mma_bf16_16816(o[2 * dp], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b0, b1);
          mma_bf16_16816(o[2 * dp + 1], pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3], b2, b3);
        }
      }
    }
  };

  bool failed = false;
  int lt = 0;
  for (; lt < n_pref; ++lt) {
    const int st = lt % kStages;
    const uint32_t par = (lt / kStages) & 1;
    if (tid == 0) sh_ok = mbar_wait_bounded(bar0 + 8 * st, par) ? 1 : 0;
    __syncthreads();
    if (!sh_ok) {
      failed = true;
      break;
    }
    mbar_try_wait(bar0 + 8 * st, par);
    const int kb = (t0 + lt) * kTile;
    if (kb + kTile > P) {  // last prefix tile: zero V rows past the prefix (unwritten memory may be NaN)
      uint8_t* v = smem + st * kStageBytes + 2 * kHalfBytes;
      for (int e = tid; e < kTile * 16; e += kWarps * 32) {
        const int row = e >> 4, hf = (e >> 3) & 1;
        if (kb + row >= P) *reinterpret_cast<uint4*>(v + hf * kHalfBytes + row * 128 + (e & 7) * 16) =
                               make_uint4(0, 0, 0, 0);
      }
      __syncthreads();
    }
    tile(st, false, kb);
    __syncthreads();
    if (tid == 0 && lt + kStages < n_pref) {
      fence_proxy_async_smem();
      issue(lt + kStages, st);
    }
  }
  if (failed) {
    if (tid == 0) {
      record_error(c.status, RESA_DEV_WAIT_TIMEOUT, bh);
      for (int k = lt; k < min(n_pref, lt + kStages); ++k)
        mbar_wait_bounded(bar0 + 8 * (k % kStages), (k / kStages) & 1);
    }
    return;
  }
  // causal tail from k_new / v_new (written into stage 0 with the TMA layout)
  for (int tt = 0; tt < n_tail; ++tt) {
    const int tb = tt * kTile;
    uint8_t* kst = smem;
    uint8_t* vst = smem + 2 * kHalfBytes;
    for (int e = tid; e < kTile * 16; e += kWarps * 32) {
      const int row = e >> 4, ch = e & 15;
      const int t = tb + row;
      uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
      if (t < f) {
        const size_t src = ((static_cast<size_t>(b) * f + t) * c.Hkv + h) * kHeadDim + ch * 8;
        kv = *reinterpret_cast<const uint4*>(a.k_new + src);
        vv = *reinterpret_cast<const uint4*>(a.v_new + src);
      }
      const uint32_t off = (ch >> 3) * kHalfBytes + sw128(row, ch & 7);
      *reinterpret_cast<uint4*>(kst + off) = kv;
      *reinterpret_cast<uint4*>(vst + off) = vv;
    }
    __syncthreads();
    tile(0, true, tb);
    __syncthreads();
  }

  // epilogue: normalised partial O and log2-sum-exp per row
#pragma unroll
  for (int x = 1; x < 4; x <<= 1) {
    lA += __shfl_xor_sync(0xffffffffu, lA, x);
    lB += __shfl_xor_sync(0xffffffffu, lB, x);
  }
  const float invA = lA > 0.f ? 1.f / lA : 0.f, invB = lB > 0.f ? 1.f / lB : 0.f;
#pragma unroll
  for (int hf = 0; hf < 2; ++hf) {
    const int r = hf ? rB : rA;
    const int i = hf ? iB : iA;
    if (i < 0) continue;
    const size_t prow = (static_cast<size_t>(b) * f + i) * c.Hq + h * g + r % g;
    float* dst = a.o_part + (prow * a.splits + s) * kHeadDim;
    const float inv = hf ? invB : invA;
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) {
      const int d = 8 * nt + 2 * (lane & 3);
      *reinterpret_cast<float2*>(dst + d) = make_float2(o[nt][2 * hf] * inv, o[nt][2 * hf + 1] * inv);
    }
    if ((lane & 3) == 0) {
      const float l = hf ? lB : lA, m = hf ? mB : mA;
      a.lse_part[prow * a.splits + s] = l > 0.f ? m + log2f(l) : kNegInf;
    }
  }
}

}  // namespace

int rectify_row_groups(int g, int f) { return (g * f + kRows - 1) / kRows; }

cudaError_t launch_rectify(const CacheView& c, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                           const uint16_t* q_new, const uint16_t* k_new, const uint16_t* v_new, int f,
                           float sm_scale, int splits, float* o_part, float* lse_part, cudaStream_t st) {
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(rectify_kernel), kSmem, 1);
  if (e != cudaSuccess) return e;
  RectArgs a{q_new, k_new, v_new, f, splits, sm_scale * 1.44269504088896340736f, o_part, lse_part};
  const dim3 grid(splits, rectify_row_groups(c.g, f), c.B * c.Hkv);
  return launch_pdl(rectify_kernel, grid, dim3(kWarps * 32), kSmem, st, tm_k, tm_v, c, a);
}

}  // namespace resa
