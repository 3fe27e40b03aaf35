// Dense rectification attention (Section 2.2; Algorithm 1 DenseForward) on
// the 5th-generation tensor cores (tcgen05, accumulators in tensor memory).
//
// Work: for each (sequence b, KV head h) the f most recent tokens' queries of
// the group attend causally to the cache: query row i (position T - f + i)
// sees positions [0, T - f + i]. Keys/values of the prefix [0, T - f) come
// from the paged cache, those of the f tokens from k_new / v_new.
//
// Rows: r = 8 * i + j (token i, query head h*g + j; heads padded to 8, so for
// g = 7 the M-tile count f/16 is the same as unpadded). A CTA owns up to two
// 128-row M-tiles (256 rows) of one (b, h) and a contiguous range of 64-key
// tiles (a key split); the last split also takes the causal tail. Partials
// (normalised O, log2-sum-exp) are combined by merge_kernel.
//
// CTA = 12 warps:
//   warps 0, 2, 3  TMA producers: 64-key K and V tiles of the prefix, one
//               SWIZZLE_128B box per 16-key page per 64-column half (16 per
//               tile, spread over the three warps: copies issued by the lanes
//               of one warp go out one after another), into a 5-stage ring
//               (kv_full / kv_empty mbarriers); page ids are read 32 blocks at
//               a time. The tiles of the f new tokens come from k_new / v_new
//               by 4-D TMA boxes (64 tokens x 64 dims of one head), only up to
//               the last token of the CTA's rows (later keys are causally
//               masked).
//   warp 1      allocates 512 TMEM columns; lane 0 issues the MMAs:
//               S[t] = Q K^T (M 128, N 64, K 128; both operands K-major from
//               shared memory) into a double-buffered TMEM S, and
//               O += P V (M 128, N 128, K 64) with P read from tensor memory
//               (the A operand) and V an MN-major shared-memory operand.
//   warps 4-11  softmax: one thread per query row (TMEM lane), so the row max
//               and sum need no shuffles. P (bf16, key pairs packed per
//               column) is stored over the first 32 columns of its own S tile,
//               so no shared memory or wait on the previous PV is needed; S of
//               tile t + 2 is issued only after PV of tile t has read that P.
//               O is rescaled in TMEM only when a row maximum grows by more
//               than 2^8 (exact: the exponent base is carried along).
// TMEM columns: O[mt] = [128 mt, 128 mt + 128), S/P[buf][mt] = 256 + 64 (2 buf + mt).
// Every mbarrier wait is bounded; a wait that runs out records
// RESA_DEV_WAIT_TIMEOUT and the CTA winds down, freeing its TMEM.
#include "resa_device.cuh"
#include "resa_launch.h"

namespace resa {
namespace {

constexpr int kThreads = 384;
constexpr int kSoftmaxWarp0 = 4;
constexpr int kMTile = 128;
constexpr int kMaxMTiles = 2;
constexpr int kRowsPerCta = kMTile * kMaxMTiles;  // 256
constexpr int kTileKeys = 64;
constexpr int kStages = 5;
constexpr int kQHalf = kRowsPerCta * 128;          // [256 rows][64 dims] bf16 = 32 KB
constexpr int kKVHalf = kTileKeys * 128;           // [64 keys][64 dims] = 8 KB
constexpr int kStageBytes = 4 * kKVHalf;           // K (2 halves) + V (2 halves) = 32 KB
constexpr int kQTile = kMTile * 128;               // one M-tile of one Q half = 16 KB
constexpr int kOffQ = 0;
constexpr int kOffKV = 2 * kQHalf;                       // 64 KB
constexpr int kOffBar = kOffKV + kStages * kStageBytes;  // 224 KB
constexpr int kSmem = kOffBar + 256 + 1024;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColO = 0;
constexpr uint32_t kColS = 256;
constexpr uint32_t kIdescS = idesc_bf16_f32(kMTile, kTileKeys, 0, 0);
constexpr uint32_t kIdescO = idesc_bf16_f32(kMTile, 128, 0, 1);
constexpr float kRescaleLog2 = 8.f;
constexpr float kNegInf = -__builtin_huge_valf();

// barrier slots (uint64) in the barrier region
constexpr int kBarKvFull = 0, kBarKvEmpty = kStages, kBarSFull = 2 * kStages, kBarPFull = kBarSFull + 2,
              kBarODone = kBarPFull + 2, kBarFinal = kBarODone + 2;
constexpr int kTmemSlot = 240;  // byte offset of the TMEM base address in the barrier region
static_assert(8 * (kBarFinal + 1) <= kTmemSlot, "barriers overlap the TMEM address slot");

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

// Warp-uniform bounded wait: lane 0 polls, the verdict is broadcast, and every
// lane then observes the completed phase itself.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait_bounded(bar, parity) ? 1 : 0;
  ok = __shfl_sync(0xffffffffu, ok, 0);
  if (ok) mbar_try_wait(bar, parity);
  return ok != 0;
}

__global__ void __launch_bounds__(kThreads, 1) rectify_kernel(const __grid_constant__ CUtensorMap tm_k,
                                                              const __grid_constant__ CUtensorMap tm_v,
                                                              const __grid_constant__ CUtensorMap tm_kn,
                                                              const __grid_constant__ CUtensorMap tm_vn,
                                                              CacheView c, RectArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + kOffBar;
  auto bar = [&](int slot) -> uint32_t { return bar0 + 8u * slot; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + kOffBar + kTmemSlot);

  const int s = blockIdx.x, rg = blockIdx.y, bh = blockIdx.z;
  const int b = bh / c.Hkv, h = bh % c.Hkv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int f = a.f, g = c.g;
  const int rows_total = 8 * f;
  const int row0 = rg * kRowsPerCta;
  const int MT = min(kMaxMTiles, (rows_total - row0 + kMTile - 1) / kMTile);

  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(bar(kBarKvFull + i), 1);
      mbar_init(bar(kBarKvEmpty + i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(kBarSFull + i), 1);
      mbar_init(bar(kBarPFull + i), kMTile * MT);
      mbar_init(bar(kBarODone + i), 1);
    }
    mbar_init(bar(kBarFinal), 1);
    fence_mbar_init();
    prefetch_tmap(&tm_k);
    prefetch_tmap(&tm_v);
    prefetch_tmap(&tm_kn);
    prefetch_tmap(&tm_vn);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_launch_dependents();
  pdl_wait();

  const bool inactive = c.active != nullptr && c.active[b] == 0;  // left out: no work, no output row
  const int T = inactive ? f : c.seq_lens[b];
  const bool bad = inactive || (T < f || T > c.max_blocks * kBlock);
  const int P = T - f;  // prefix keys from the cache
  const int ntp = bad ? 0 : (P + kTileKeys - 1) / kTileKeys;
  const int per = (ntp + a.splits - 1) / a.splits;
  const int t0 = s * per;
  const int n_pref = max(0, min(ntp, t0 + per) - t0);
  // tail tiles of the f new tokens, up to the last token of this CTA's rows
  // (later keys are causally masked for every row here)
  const int tok_end = min(f, (row0 + MT * kMTile + 7) / 8);
  const int n_tail = (!bad && s == a.splits - 1) ? (tok_end + kTileKeys - 1) / kTileKeys : 0;
  const int n_tiles = n_pref + n_tail;
  if (bad && !inactive && tid == 0 && s == 0 && rg == 0) record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);

  // Q tile: rows row0 .. row0 + 128 MT - 1, zero for padding rows
  for (int e0 = 0; e0 < MT * kMTile * 16; e0 += 4 * kThreads) {  // four loads in flight per thread
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int e = e0 + u * kThreads + tid;
      const int row = e >> 4, ch = e & 15;
      const int rr = row0 + row, i = rr >> 3, j = rr & 7;
      v[u] = make_uint4(0, 0, 0, 0);
      if (e < MT * kMTile * 16 && !bad && i < f && j < g)
        v[u] = *reinterpret_cast<const uint4*>(a.q_new + ((static_cast<size_t>(b) * f + i) * c.Hq + h * g + j) *
                                                             kHeadDim + ch * 8);
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int e = e0 + u * kThreads + tid;
      const int row = e >> 4, ch = e & 15;
      if (e < MT * kMTile * 16)
        *reinterpret_cast<uint4*>(smem + kOffQ + (ch >> 3) * kQHalf + sw128(row, ch & 7)) = v[u];
    }
  }
  fence_proxy_async_smem();
  __syncthreads();

  if (warp == 0 || warp == 2 || warp == 3) {
    // ------------------------------------------------------ producers ---
    // Three warps issue the boxes of each tile (TMA copies issued by the
    // lanes of one warp go out one after another; separate warps issue in
    // parallel): box j of a prefix tile (page j / 4, part j % 4: K or V, one
    // 64-column half) is issued by producer j % 3; warp 0 also posts the
    // stage's byte count. Page rows of the prefix blocks are read 32 at a
    // time (eight tiles).
    const int pw = warp == 0 ? 0 : warp - 1;  // producer 0, 1, 2
    int win = -1, my_row = -1;
    for (int t = 0; t < n_tiles; ++t) {
      const int st = t % kStages;
      if (t >= kStages && !warp_wait(bar(kBarKvEmpty + st), ((t / kStages) - 1) & 1)) {
        if (lane == 0) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, bh);
        break;
      }
      const uint32_t kdst = sbase + kOffKV + st * kStageBytes;
      if (t < n_pref) {
        if ((t & ~7) != win) {
          win = t & ~7;
          const int blk = (t0 + win) * (kTileKeys / kBlock) + lane;
          my_row = -1;
          if (blk * kBlock < P) {
            const int page = c.page_table[static_cast<size_t>(b) * c.max_blocks + blk];
            if (page >= 0 && page < c.num_pages)
              my_row = (page * c.Hkv + h) * kBlock;
            else if (pw == 0 && win * (kTileKeys / kBlock) + lane < n_pref * (kTileKeys / kBlock))
              record_error(c.status, RESA_DEV_PAGE_RANGE, b);  // a block this CTA uses: left out
          }
        }
        const int slot = (t - win) * (kTileKeys / kBlock);
        if (pw == 0) {
          int pages = 0;
#pragma unroll
          for (int pg = 0; pg < kTileKeys / kBlock; ++pg) pages += __shfl_sync(0xffffffffu, my_row, slot + pg) >= 0 ? 1 : 0;
          if (lane == 0) mbar_arrive_expect_tx(bar(kBarKvFull + st), pages * 4 * 2048);
        }
        // this producer's boxes j = pw + 3 l (lane l), j < 16
        const int j = pw + 3 * lane;
        const int row = __shfl_sync(0xffffffffu, my_row, slot + ((j >> 2) & 3));
        if (j < 16 && row >= 0) {
          const int part = j & 3;
          tma_load_2d_stream(kdst + part * kKVHalf + (j >> 2) * 2048, part < 2 ? &tm_k : &tm_v, bar(kBarKvFull + st),
                      (part & 1) * 64, row);
        }
      } else {
        // tail tile: tokens tb .. tb + 63 of the f new ones, by TMA from
        // k_new / v_new viewed as [B][f][Hkv][128] (tokens >= f read as zero);
        // producer pw issues boxes pw and (pw == 0) 3
        const int tb = (t - n_pref) * kTileKeys;
        if (lane == 0) {
          if (pw == 0) mbar_arrive_expect_tx(bar(kBarKvFull + st), 4 * kKVHalf);
          for (int part = pw; part < 4; part += 3)
            tma_load_4d(kdst + part * kKVHalf, part < 2 ? &tm_kn : &tm_vn, bar(kBarKvFull + st), (part & 1) * 64, h,
                        tb, b);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA ---
    if (lane == 0) {
      // Base descriptors; an MMA's operand is base + (byte offset >> 4) (the
      // 14-bit start-address field cannot carry: shared memory is < 256 KB).
      const uint64_t dq = smem_desc_sw128(sbase + kOffQ, 16, 1024);
      const uint64_t dkv = smem_desc_sw128(sbase + kOffKV, 16, 1024);
      const uint64_t dvv = smem_desc_sw128(sbase + kOffKV + 2 * kKVHalf, kKVHalf, 1024);
      auto issue_pv = [&](int u) -> bool {
        const int bu = u & 1, su = u % kStages;
        if (!mbar_wait_bounded(bar(kBarPFull + bu), (u >> 1) & 1)) return false;
        tc_fence_after();
        const uint64_t dv = dvv + ((su * kStageBytes) >> 4);
        for (int mt = 0; mt < MT; ++mt) {
          // P of (u, mt) sits in the first 32 columns of S[bu][mt], 8 columns per 16 keys
          const uint32_t ptmem = tmem + kColS + (bu * kMaxMTiles + mt) * kTileKeys;
          for (int kk = 0; kk < kTileKeys / 16; ++kk)
            umma_bf16_tmem_a(tmem + kColO + mt * 128, ptmem + kk * 8, dv + ((kk * 2048) >> 4), kIdescO,
                             (u > 0 || kk > 0) ? 1u : 0u);
        }
        umma_commit(bar(kBarODone + bu));
        umma_commit(bar(kBarKvEmpty + su));
        return true;
      };
      bool ok = true;
      for (int t = 0; t < n_tiles && ok; ++t) {
        const int st = t % kStages, buf = t & 1;
        if (!mbar_wait_bounded(bar(kBarKvFull + st), (t / kStages) & 1)) {
          ok = false;
          break;
        }
        // S(t) overwrites S[buf], whose first columns hold P(t - 2): PV(t - 2) must be done
        if (t >= 2 && !mbar_wait_bounded(bar(kBarODone + buf), ((t - 2) >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t dk = dkv + ((st * kStageBytes) >> 4);
        for (int mt = 0; mt < MT; ++mt) {
          for (int ks = 0; ks < 8; ++ks) {
            const uint32_t off = (ks & 3) * 32;
            umma_bf16(tmem + kColS + (buf * kMaxMTiles + mt) * kTileKeys,
                      dq + (((ks >> 2) * kQHalf + mt * kQTile + off) >> 4),
                      dk + (((ks >> 2) * kKVHalf + off) >> 4), kIdescS, ks > 0 ? 1u : 0u);
          }
        }
        umma_commit(bar(kBarSFull + buf));
        if (t >= 1) ok = issue_pv(t - 1);
      }
      if (ok && n_tiles > 0) ok = issue_pv(n_tiles - 1);
      if (!ok) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, bh);
      // let every issued MMA finish before the CTA may free its TMEM
      umma_commit(bar(kBarFinal));
      mbar_wait_bounded(bar(kBarFinal), 0);
    }
    __syncwarp();
  } else if (warp >= kSoftmaxWarp0) {
    // -------------------------------------------------------- softmax ---
    const int mt = (warp - kSoftmaxWarp0) >> 2, quarter = warp & 3;
    const int rit = quarter * 32 + lane;  // row within the M-tile = TMEM lane
    const int rr = row0 + mt * kMTile + rit;
    const int ti = rr >> 3, tj = rr & 7;
    const bool valid_row = ti < f && tj < g;
    const int sm_tid = (warp - kSoftmaxWarp0) * 32 + lane;  // 0 .. 128 MT - 1
    if (mt < MT) {
      const uint32_t lane_base = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
      float m_used = kNegInf, l = 0.f;
      bool ok = true;
      for (int t = 0; t < n_tiles; ++t) {
        const int buf = t & 1, st = t % kStages;
        if (!warp_wait(bar(kBarSFull + buf), (t >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        float sv[kTileKeys];  // raw scores q.k of this row
        {
          uint32_t r0[32], r1[32];
          const uint32_t col = kColS + (buf * kMaxMTiles + mt) * kTileKeys;
          tmem_ld32(lane_base + col, r0);
          tmem_ld32(lane_base + col + 32, r1);
          tmem_ld_wait();
#pragma unroll
          for (int x = 0; x < 32; ++x) {
            sv[x] = __uint_as_float(r0[x]);
            sv[32 + x] = __uint_as_float(r1[x]);
          }
        }
        const bool tail = t >= n_pref;
        const int kb = tail ? (t - n_pref) * kTileKeys : (t0 + t) * kTileKeys;
        const int lim = tail ? min(f - 1 - kb, ti - kb) : P - 1 - kb;  // key c visible iff c <= lim
        if (lim < kTileKeys - 1) {
#pragma unroll
          for (int x = 0; x < kTileKeys; ++x) sv[x] = (x <= lim) ? sv[x] : kNegInf;
        }
        float mx;
        {
          // three-input maxima, four independent chains of 16 keys
          float m4[4];
#pragma unroll
          for (int y = 0; y < 4; ++y) {
            float v = sv[y];
            static_assert(kTileKeys == 64, "keys y, y + 4, ..., y + 60");
#pragma unroll
            for (int k = 0; k < 7; ++k) v = max3f(v, sv[y + 4 + 8 * k], sv[y + 8 + 8 * k]);
            m4[y] = fmaxf(v, sv[y + 60]);
          }
          mx = fmaxf(max3f(m4[0], m4[1], m4[2]), m4[3]) * a.scale_log2;  // scale > 0 keeps the order
        }
        const float m_new = fmaxf(m_used, mx);
        const bool need = m_new > m_used + kRescaleLog2;  // per row
        const bool scale_o = need && t >= 1 && m_used != kNegInf;
        // The O rescale is warp-collective (tcgen05.ld/st are .sync.aligned):
        // the whole warp takes it if any of its rows needs it (rows that do
        // not keep alpha = 1), once PV of tile t - 1 has landed.
        if (__any_sync(0xffffffffu, scale_o)) {
          if (!warp_wait(bar(kBarODone + ((t - 1) & 1)), ((t - 1) >> 1) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const float alpha = scale_o ? exp2f(m_used - m_new) : 1.f;
          for (int ch = 0; ch < 4; ++ch) {
            uint32_t r[32];
            tmem_ld32(lane_base + kColO + mt * 128 + ch * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int x = 0; x < 32; ++x) r[x] = __float_as_uint(__uint_as_float(r[x]) * alpha);
            tmem_st32(lane_base + kColO + mt * 128 + ch * 32, r);
          }
          tmem_st_wait();
          l *= alpha;
        }
        if (need) m_used = m_new;
        const float nbase = -safe_base(m_used);
        uint32_t w[kTileKeys / 2];  // P row as packed bf16 pairs (keys 2x, 2x + 1)
        // exponent arguments and row sums two keys per instruction
        const uint64_t sc2 = pack_f32x2(a.scale_log2, a.scale_log2), nb2 = pack_f32x2(nbase, nbase);
        uint64_t ls2[2] = {0ull, 0ull};
#pragma unroll
        for (int x = 0; x < kTileKeys / 2; ++x) {
          float x0, x1;
          unpack_f32x2(fma_f32x2(pack_f32x2(sv[2 * x], sv[2 * x + 1]), sc2, nb2), x0, x1);
          const float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
          ls2[x & 1] = add_f32x2(ls2[x & 1], pack_f32x2(p0, p1));
          w[x] = pack_bf16x2(p0, p1);
        }
        {
          float a0, a1, b0, b1;
          unpack_f32x2(ls2[0], a0, a1);
          unpack_f32x2(ls2[1], b0, b1);
          l += (a0 + a1) + (b0 + b1);
        }
        // P over the S columns it came from (this thread's lane; S is in registers)
        tmem_st32(lane_base + kColS + (buf * kMaxMTiles + mt) * kTileKeys, w);
        tmem_st_wait();
        if (!tail && kb + kTileKeys > P) {
          // keys past the prefix may sit in unwritten memory: zero their V rows
          uint8_t* v = smem + kOffKV + st * kStageBytes + 2 * kKVHalf;
          const int first = max(0, P - kb);
          for (int e = sm_tid; e < (kTileKeys - first) * 16; e += kMTile * MT) {
            const int row = first + (e >> 4), hf = (e >> 3) & 1;
            *reinterpret_cast<uint4*>(v + hf * kKVHalf + row * 128 + (e & 7) * 16) = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();  // generic stores, read next by the tensor core
        }
        tc_fence_before();
        mbar_arrive(bar(kBarPFull + buf));
      }
      if (!ok && lane == 0) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, bh);
      // ---- epilogue: normalised partial O and log2-sum-exp of this row ----
      const bool have = ok && n_tiles > 0 &&
                        warp_wait(bar(kBarODone + ((n_tiles - 1) & 1)), ((n_tiles - 1) >> 1) & 1);
      if (have) tc_fence_after();
      const float inv = (have && l > 0.f) ? 1.f / l : 0.f;
      const size_t prow_g = (static_cast<size_t>(b) * f + ti) * c.Hq + h * g + tj;
      float* dst = a.o_part + (prow_g * a.splits + s) * kHeadDim;
      for (int ch = 0; ch < 4; ++ch) {
        uint32_t r[32];
        if (have) {
          tmem_ld32(lane_base + kColO + mt * 128 + ch * 32, r);
          tmem_ld_wait();
        }
        if (valid_row && !bad) {
#pragma unroll
          for (int x = 0; x < 32; x += 4)
            *reinterpret_cast<float4*>(dst + ch * 32 + x) =
                have ? make_float4(__uint_as_float(r[x]) * inv, __uint_as_float(r[x + 1]) * inv,
                                   __uint_as_float(r[x + 2]) * inv, __uint_as_float(r[x + 3]) * inv)
                     : make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      if (valid_row && !bad) a.lse_part[prow_g * a.splits + s] = (have && l > 0.f) ? m_used + log2f(l) : kNegInf;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

int rectify_row_groups(int g, int f) {
  (void)g;
  return (8 * f + kRowsPerCta - 1) / kRowsPerCta;
}

cudaError_t launch_rectify(const CacheView& c, const CUtensorMap& tm_k, const CUtensorMap& tm_v,
                           const CUtensorMap& tm_kn, const CUtensorMap& tm_vn, const uint16_t* q_new,
                           const uint16_t* k_new, const uint16_t* v_new, int f, float sm_scale, int splits,
                           float* o_part, float* lse_part, cudaStream_t st) {
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(rectify_kernel), kSmem, 1);
  if (e != cudaSuccess) return e;
  RectArgs a{q_new, k_new, v_new, f, splits, sm_scale * 1.44269504088896340736f, o_part, lse_part};
  const dim3 grid(splits, rectify_row_groups(c.g, f), c.B * c.Hkv);
  return launch_pdl(rectify_kernel, grid, dim3(kThreads), kSmem, st, tm_k, tm_v, tm_kn, tm_vn, c, a);
}

}  // namespace resa
