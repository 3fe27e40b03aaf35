// Block selection (Section 2.1 "Block Selection"; Eq. 4 and Eq. 5).
//
// score_kernel  persistent, one CTA per SM: each of its 16 warps streams 6 KB
//               (small caches: 4 KB) pieces of the block summaries with its
//               own bulk copies through its own shared-memory ring and
//               scores them with the pooled query of the piece's GQA group
//               (mean of the g heads, fp32); eight lanes take one block, a
//               lane 16 dims of k_min and k_max, and the 128-dim sum is a
//               fixed-order butterfly over the 8 lanes.
// top-n        one CTA (caches of up to kTopnCtaMaxBlocks blocks per
//               sequence) or one 8-CTA cluster (larger caches) per (sequence,
//               KV head). The n of Eq. 5 is evaluated on the device from the
//               device-resident length. The last n_local blocks are always
//               taken (score +inf); the rest of the budget is the largest
//               order-preserving keys of the other blocks, found by a radix
//               select over key - min key with 8-bit digits from the top
//               significant bit of the unit's key range (keys staged in shared
//               memory; in the cluster form every exchange between the CTAs,
//               extremes, histograms and counts, is stored into the other
//               CTAs' shared memory by stores that complete on the
//               receiver's mbarrier). The selected
//               ids are written in ascending order by a ballot compaction that
//               resolves ties at the threshold toward the lower block index.
//
// Both top-n kernels read the length and evaluate Eq. 5 before waiting on the
// score kernel: that kernel lets its dependents launch only after its own wait
// on the preceding kernel (the append commit, or the previous fused step's
// merge, that advances the length) has returned, and the length is read from
// L2.

#include "resa_device.cuh"
#include "resa_launch.h"

namespace resa {
namespace {

constexpr int kTopnCluster = 8;                                   // CTAs per (sequence, KV head)
constexpr int kTopnThreads = 512;
constexpr int kTopnWarps = kTopnThreads / 32;
constexpr int kTopnSmemMax = 200 * 1024;                           // staged keys per CTA, bytes
constexpr int kTopnCtaThreads = 512;                                // one-CTA form
constexpr int kTopnCtaWarps = kTopnCtaThreads / 32;
constexpr int kTopnCtaMaxBlocks = 6144;  // the one-CTA form serves caches up to this many blocks per sequence
constexpr int kTopnCtaKeys = kTopnCtaMaxBlocks / kTopnCtaThreads;   // keys held per thread
static_assert(kTopnCtaKeys * kTopnCtaThreads == kTopnCtaMaxBlocks && kTopnCtaKeys <= 32, "one-CTA key layout");

// Eq. 4 partial sum over 8 dims, accumulated into s. Since k_min <= k_max in
// every dimension, max(q k_max, q k_min) is q k_max where q >= 0 and q k_min
// where q < 0 (sign bit set): one byte permute per bf16 pair picks the factor
// (`sel`, from the signs of the pooled query), and one fp32 FMA per dimension
// accumulates q times it. The product is the one the max would return, bit
// for bit (infinities and a zero q included); a NaN key makes both k_min and
// k_max NaN in its dimension, so the picked factor is NaN either way.
__device__ __forceinline__ float quest_term8(const float* qf, const uint32_t* sel, const uint4& mn, const uint4& mx,
                                             float s) {
  const uint32_t a[4] = {mn.x, mn.y, mn.z, mn.w};
  const uint32_t c[4] = {mx.x, mx.y, mx.z, mx.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t m = __byte_perm(a[i], c[i], sel[i]);
    s = fmaf(qf[2 * i], bf16_lo(m), s);
    s = fmaf(qf[2 * i + 1], bf16_hi(m), s);
  }
  return s;
}

// __byte_perm selector for one bf16 pair (low element first): bytes of k_min
// (0-3) where the query element's sign bit is set, of k_max (4-7) elsewhere.
__device__ __forceinline__ uint32_t quest_selector(float q_lo, float q_hi) {
  const uint32_t lo = signbit(q_lo) ? 0x0010u : 0x0054u;
  const uint32_t hi = signbit(q_hi) ? 0x3200u : 0x7600u;
  return lo | hi;
}

// Persistent score kernel: one CTA per SM. The (sequence, KV head) units'
// summaries are cut into pieces of kPieceBlocks blocks (contiguous); CTA x
// owns the piece range [x * per, (x + 1) * per) of the flattened piece list
// and its warp w takes every 16th piece of it (w, w + 16, ...). Each warp
// streams its pieces with 1-D bulk copies issued by its own lane 0 through
// its own kScoreStages-stage shared-memory ring: copies issued by one thread
// complete one after another, so sixteen independent issuers keep enough
// bytes in flight per SM. Every stage is filled before the dependency wait,
// and a warp refills a stage as soon as it has scored it (lane 0 locates the
// refill's piece while it waits for the stage's copy). Two shapes, the same 192 KB of rings: 12-block
// (6 KB) pieces in 2 stages when the cache has at least one such piece per
// warp of the grid (measured: they beat 8 blocks in 3 stages, and 16 blocks
// with 12 warps, at 32K x 8 and 256K x 1), else 8-block (4 KB) pieces in 3
// stages, which give more warps a piece. Eight lanes score one block, a lane
// 16 dims of k_min and k_max (two 16-byte chunks, dims 8c..8c+7 and
// 64+8c..64+8c+7 for lane c of the eight), and the 128-dim sum ends in a
// fixed-order 8-lane butterfly.
constexpr int kScoreWarps = 16;
constexpr int kMaxBatch = 1024;  // sequences per call supported by the score kernel
constexpr int score_piece_bytes(int piece_blocks) { return piece_blocks * 2 * kHeadDim * 2; }
constexpr int score_ring_bytes(int piece_blocks, int stages) {
  return kScoreWarps * stages * score_piece_bytes(piece_blocks);
}
// rings and their barriers; the per-sequence tables (score_table_bytes) follow
constexpr int score_smem_bytes(int piece_blocks, int stages) {
  return score_ring_bytes(piece_blocks, stages) + kScoreWarps * stages * 8;
}
constexpr int score_table_bytes(int B) { return (3 * B + 1) * static_cast<int>(sizeof(int)); }

// At most 88 registers: a score CTA (512 x 88) then fits beside one merge
// CTA (256 x 64), so that one launched early issues its first copies while
// the preceding step's merge runs, and a top-n cluster CTA launched early
// (512 x 40) fits beside a score CTA.
template <int kPieceBlocks, int kScoreStages>
__global__ void __maxnreg__(88) score_kernel(CacheView c, const uint16_t* __restrict__ q,
                                                                    float* __restrict__ scores) {
  static_assert(kPieceBlocks % 4 == 0, "four lane groups score a piece's blocks four at a time");
  constexpr int kPieceBytes = score_piece_bytes(kPieceBlocks);
  constexpr int kScoreRing = score_ring_bytes(kPieceBlocks, kScoreStages);
  constexpr int kScoreSmem = score_smem_bytes(kPieceBlocks, kScoreStages);
  extern __shared__ __align__(1024) uint8_t smem[];
  // per-sequence block counts and the piece prefix over (sequence, head)
  // units, after the rings and their barriers (sized by the batch, so that
  // the top-n CTAs launched early fit beside this CTA)
  int* sh_M = reinterpret_cast<int*>(smem + kScoreSmem);
  int* sh_T = sh_M + c.B;
  int* sh_pref = sh_T + c.B;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  uint8_t* ring = smem + warp * kScoreStages * kPieceBytes;
  const uint32_t ring_s = smem_u32(ring);
  const uint32_t bar0 = smem_u32(smem) + kScoreRing + warp * kScoreStages * 8;
  if (lane == 0) {
    for (int i = 0; i < kScoreStages; ++i) mbar_init(bar0 + 8 * i, 1);
    fence_mbar_init();
  }
  // per-sequence block counts and the exclusive prefix of Hkv * pieces-per-head
  // over sequences (lengths out of range count as empty: top-n reports them)
  auto build_tables = [&]() {
    for (int b = tid; b < c.B; b += blockDim.x) {
      const int T = __ldcg(c.seq_lens + b) + c.pending;
      const bool bad = T < 0 || T > c.max_blocks * kBlock;
      sh_M[b] = bad ? 0 : (T + kBlock - 1) / kBlock;
      sh_T[b] = bad ? 0 : T;
    }
    __syncthreads();
    if (warp == 0) {
      int carry = 0;
      for (int b0 = 0; b0 < c.B; b0 += 32) {
        const int b = b0 + lane;
        const int v = b < c.B ? c.Hkv * ((sh_M[b] + kPieceBlocks - 1) / kPieceBlocks) : 0;
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
  };
  // piece index -> (sequence, head, first block, blocks): binary search of the prefix
  auto locate = [&](int pi, int& b, int& h, int& blk0, int& nblk) {
    int lo = 0, hi = c.B - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (sh_pref[mid] <= pi) lo = mid;
      else hi = mid - 1;
    }
    b = lo;
    const int M = sh_M[b];
    const int per_head = (M + kPieceBlocks - 1) / kPieceBlocks;
    const int r = pi - sh_pref[b];
    h = r / per_head;
    blk0 = (r % per_head) * kPieceBlocks;
    nblk = min(kPieceBlocks, M - blk0);
  };
  // The first pieces are fetched before the wait for the preceding kernel:
  // every earlier writer of the summaries has completed by the time this
  // kernel starts. The commits and the bulk summary build let their dependents
  // launch only at exit, and this kernel (whose append writes them in a fused
  // step) is always followed by a top-n kernel that lets its own dependents
  // launch only after its wait. The lengths may still change under this
  // prologue (the merge of a fused decode step advances them after letting
  // its dependents launch), so they are read again after the wait, and if a
  // block count differs the warps drain their copies and start over.
  build_tables();
  int total, per, c0, ncta, nmine, kbase = 0;  // kbase: copies issued before the current piece list
  auto my_range = [&]() {
    total = sh_pref[c.B];
    per = (total + gridDim.x - 1) / gridDim.x;
    c0 = blockIdx.x * per;
    ncta = max(0, min(total, c0 + per) - c0);
    nmine = ncta > warp ? (ncta - warp + kScoreWarps - 1) / kScoreWarps : 0;
  };
  my_range();
  // the location (sequence, head, first block, blocks) of the piece in each
  // stage, written by lane 0 when it issues the copy and read by the warp
  // when it scores the stage, so that a piece is located once
  __shared__ int4 sh_loc[kScoreWarps][kScoreStages];
  struct Src {
    const uint16_t* p;
    uint32_t bytes;
    int4 loc;
  };
  auto piece_src = [&](int k) {  // this warp's k-th piece: its summaries, size and location
    int b, h, blk0, nblk;
    locate(c0 + warp + k * kScoreWarps, b, h, blk0, nblk);
    return Src{c.summ + ((static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks + blk0) * 2 * kHeadDim,
               static_cast<uint32_t>(nblk) * 2 * kHeadDim * 2, make_int4(b, h, blk0, nblk)};
  };
  auto issue_src = [&](int k, const Src& src) {  // lane 0: piece k into stage (kbase + k) % kScoreStages
    const int stage = (kbase + k) % kScoreStages;
    const uint32_t bar = bar0 + 8 * stage;
    sh_loc[warp][stage] = src.loc;
    mbar_arrive_expect_tx(bar, src.bytes);
    bulk_load_stream(ring_s + stage * kPieceBytes, src.p, src.bytes, bar);
  };
  auto issue = [&](int k) { issue_src(k, piece_src(k)); };
  __syncwarp();  // lane 0's barrier initialisation precedes every lane's use
  if (lane == 0)
    for (int k = 0; k < min(kScoreStages, nmine); ++k) issue(k);
  const int issued_early = min(kScoreStages, nmine);
  pdl_wait();
  pdl_launch_dependents();  // the top-n kernel reads the lengths before its own wait
  bool changed = false;
  for (int b = tid; b < c.B; b += blockDim.x) {
    const int T = __ldcg(c.seq_lens + b) + c.pending;
    const bool bad = T < 0 || T > c.max_blocks * kBlock;
    if ((bad ? 0 : (T + kBlock - 1) / kBlock) != sh_M[b]) changed = true;
    sh_T[b] = bad ? 0 : T;
  }
  if (__syncthreads_or(changed)) {
    bool drained = true;
    if (lane == 0)
      for (int k = 0; k < issued_early; ++k) drained = mbar_wait_bounded(bar0 + 8 * k, 0) && drained;
    if (!__syncthreads_and(drained)) {
      if (tid == 0) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, -1);
      return;
    }
    build_tables();
    my_range();
    kbase = issued_early;
    if (lane == 0)
      for (int k = 0; k < min(kScoreStages, nmine); ++k) issue(k);
    __syncwarp();  // the stages' locations are visible to the warp
  }

  const int ch = lane & 15, half = lane >> 4;  // the appended token: a lane folds 8 dims
  const int c8 = lane & 7, grp = lane >> 3;     // scoring: lane c8 of group grp
  int cur_unit = -1, k_fail = -1;
  float qf[16];
  uint32_t sel[8];
  uint4 ka = make_uint4(0, 0, 0, 0), va = ka;  // the appended token's key / value, this lane's 8 dims
  for (int k = 0; k < nmine; ++k) {
    const int st = (kbase + k) % kScoreStages, par = ((kbase + k) / kScoreStages) & 1;
    const int4 loc = sh_loc[warp][st];
    const int b = loc.x, h = loc.y, blk0 = loc.z, nblk = loc.w;
    const int unit = b * c.Hkv + h;
    if (unit != cur_unit) {  // pooled query (mean of the group's heads), this lane's 16 dims
      cur_unit = unit;
      if (c.pending) {
        const size_t kv = (static_cast<size_t>(b) * c.Hkv + h) * kHeadDim + ch * 8;
        ka = *reinterpret_cast<const uint4*>(c.k_append + kv);
        va = *reinterpret_cast<const uint4*>(c.v_append + kv);
      }
      // this lane's dims 8 c8 .. 8 c8 + 7 (part 0) and 64 + 8 c8 .. 64 + 8 c8 + 7
      // (part 1): lane group grp adds heads grp and grp + 4, and two butterfly
      // levels over the four groups complete the sum of the g heads
      const uint16_t* qg = q + (static_cast<size_t>(b) * c.Hq + h * c.g) * kHeadDim + c8 * 8;
      uint4 qv[4];  // head grp parts 0, 1; head grp + 4 parts 0, 1 (g <= 8)
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int head = grp + 4 * (i >> 1);
        qv[i] = head < c.g ? *reinterpret_cast<const uint4*>(qg + head * kHeadDim + 64 * (i & 1)) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int part = 0; part < 2; ++part) {
        const uint32_t w0[4] = {qv[part].x, qv[part].y, qv[part].z, qv[part].w};
        const uint32_t w1[4] = {qv[2 + part].x, qv[2 + part].y, qv[2 + part].z, qv[2 + part].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          qf[8 * part + 2 * j] = bf16_lo(w0[j]) + bf16_lo(w1[j]);
          qf[8 * part + 2 * j + 1] = bf16_hi(w0[j]) + bf16_hi(w1[j]);
        }
      }
      const float inv_g = 1.0f / static_cast<float>(c.g);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        qf[j] += __shfl_xor_sync(0xffffffffu, qf[j], 8);
        qf[j] += __shfl_xor_sync(0xffffffffu, qf[j], 16);
        qf[j] *= inv_g;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) sel[j] = quest_selector(qf[2 * j], qf[2 * j + 1]);
    }
    // lane 0 locates the piece that refills this stage before waiting for it
    const bool issue_next = lane == 0 && k + kScoreStages < nmine;
    const Src next = issue_next ? piece_src(k + kScoreStages) : Src{nullptr, 0u};
    int ok = 1;
    if (lane == 0) ok = mbar_wait_bounded(bar0 + 8 * st, par) ? 1 : 0;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    if (!ok) {
      if (lane == 0) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, unit);
      k_fail = k;
      break;
    }
    mbar_try_wait(bar0 + 8 * st, par);
    uint8_t* piece = ring + st * kPieceBytes;
    if (c.pending) {
      // Fused decode step: the appended token lands in block (T - 1) / 16.
      // The warp holding that block folds the key into its summary (Eq. 3,
      // online; a block the token opens starts empty), scores the updated
      // summary, and writes it, the key and the value to the cache.
      const int T = sh_T[b], last = (T - 1) >> 4;
      if (last >= blk0 && last < blk0 + nblk) {
        if (half == 0) {
          uint8_t* ps = piece + (last - blk0) * 512;
          float mn[8], mx[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            mn[j] = __int_as_float(0x7f800000);
            mx[j] = -__int_as_float(0x7f800000);
          }
          if (((T - 1) & (kBlock - 1)) != 0) {
            minmax8(*reinterpret_cast<const uint4*>(ps + ch * 16), mn, mx);
            minmax8(*reinterpret_cast<const uint4*>(ps + 256 + ch * 16), mn, mx);
          }
          minmax8(ka, mn, mx);
          const uint4 smin = to_bf16x8(mn), smax = to_bf16x8(mx);
          *reinterpret_cast<uint4*>(ps + ch * 16) = smin;
          *reinterpret_cast<uint4*>(ps + 256 + ch * 16) = smax;
          fence_proxy_async_smem();  // the stage is refilled by a bulk copy later
          uint16_t* sd = c.summ + summ_off(c, b, h, last);
          *reinterpret_cast<uint4*>(sd + ch * 8) = smin;
          *reinterpret_cast<uint4*>(sd + kHeadDim + ch * 8) = smax;
          const int page = c.page_table[static_cast<size_t>(b) * c.max_blocks + last];
          if (page < 0 || page >= c.num_pages) {
            if (ch == 0) record_error(c.status, RESA_DEV_PAGE_RANGE, b);
          } else {
            const size_t dst = pool_off(c, page, h, (T - 1) & (kBlock - 1)) + ch * 8;
            *reinterpret_cast<uint4*>(c.k_pool + dst) = ka;
            *reinterpret_cast<uint4*>(c.v_pool + dst) = va;
          }
        }
        __syncwarp();
      }
    }
    float* out = scores + static_cast<size_t>(unit) * c.max_blocks + blk0;
#pragma unroll
    for (int v = 0; v < kPieceBlocks / 4; ++v) {
      const int blk = 4 * v + grp;
      float sc = 0.f;
      if (blk < nblk) {
        const uint8_t* pb = piece + blk * 512 + c8 * 16;
        const uint4 mn0 = *reinterpret_cast<const uint4*>(pb), mn1 = *reinterpret_cast<const uint4*>(pb + 128);
        const uint4 mx0 = *reinterpret_cast<const uint4*>(pb + 256), mx1 = *reinterpret_cast<const uint4*>(pb + 384);
        sc = quest_term8(qf, sel, mn0, mx0, sc);
        sc = quest_term8(qf + 8, sel + 4, mn1, mx1, sc);
      }
      sc += __shfl_xor_sync(0xffffffffu, sc, 4);
      sc += __shfl_xor_sync(0xffffffffu, sc, 2);
      sc += __shfl_xor_sync(0xffffffffu, sc, 1);
      if (c8 == 0 && blk < nblk) out[blk] = sc;
    }
    __syncwarp();  // every lane has read the stage before it is refilled
    if (issue_next) {
      fence_proxy_async_smem();
      issue_src(k + kScoreStages, next);
    }
  }
  // A warp that gave up may have copies in flight (pieces k_fail .. k_fail + kScoreStages - 1):
  // wait for them (bounded) before the CTA exits.
  if (k_fail >= 0 && lane == 0) {
    for (int k2 = kbase + k_fail; k2 < kbase + min(k_fail + kScoreStages, nmine); ++k2)
      (void)mbar_wait_bounded(bar0 + 8 * (k2 % kScoreStages), (k2 / kScoreStages) & 1);
  }
}

// Order-preserving map of an fp32 score to uint32 (larger score, larger key).
// A NaN score maps to 0, below every number (-inf maps to 0x007FFFFF): NaN
// blocks rank last, among themselves by block index like every tie.
__device__ __forceinline__ uint32_t score_key(float s) {
  const uint32_t u = __float_as_uint(s);
  if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Eq. 5 for one unit: n = max(n_min, ceil(M keep)), at least n_local and at
// most M, clamped to the id row's capacity (reported). Blocks [F, M) are the
// forced local blocks (score +inf), nf of them taken; r blocks are picked
// among [0, F).
struct UnitBudget {
  int M, n, F, nf, r;
};
__device__ __forceinline__ UnitBudget unit_budget(int T, double keep, int n_min, int n_local, int n_cap,
                                                  int32_t* status, int unit, bool report) {
  UnitBudget u;
  u.M = (T + kBlock - 1) / kBlock;
  long long nn = static_cast<long long>(ceil(static_cast<double>(u.M) * keep));
  nn = max(nn, static_cast<long long>(n_min));
  nn = max(nn, static_cast<long long>(n_local));
  nn = min(nn, static_cast<long long>(u.M));
  u.n = static_cast<int>(nn);
  if (u.n > n_cap) {
    if (report) record_error(status, RESA_DEV_BUDGET_OVER_CAP, unit);
    u.n = n_cap;
  }
  u.F = u.M - min(n_local, u.M);
  u.nf = min(u.M - u.F, u.n);
  u.r = u.n - u.nf;
  return u;
}

// Warp-wide inclusive scan of one int per lane.
__device__ __forceinline__ int warp_incl_scan(int x) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  return x;
}

// The radix digit holding the rem-th largest key, from a 256-bin histogram in
// shared memory (every lane of the calling warp gets the answer): lane l owns
// digits 255-8l ... 248-8l, read as two 16-byte loads.
struct DigitPick {
  int digit, rem, whole;  // digit, rank left within it, the whole bucket is taken
};
__device__ __forceinline__ DigitPick pick_digit(const int* hist, int rem) {
  const int lane = threadIdx.x & 31;
  const int4 a0 = reinterpret_cast<const int4*>(hist)[2 * (31 - lane)];
  const int4 a1 = reinterpret_cast<const int4*>(hist)[2 * (31 - lane) + 1];
  const int cn[8] = {a1.w, a1.z, a1.y, a1.x, a0.w, a0.z, a0.y, a0.x};
  int sum = 0;
#pragma unroll
  for (int j = 0; j < 8; ++j) sum += cn[j];
  const int incl = warp_incl_scan(sum), excl = incl - sum;
  const unsigned hit = __ballot_sync(0xffffffffu, excl < rem && rem <= incl);
  const int src = hit ? __ffs(hit) - 1 : 0;  // 1 <= rem <= the histogram's total, so a lane holds it
  DigitPick p{0, 0, 0};
  if (lane == src) {
    int cum = excl;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (cum + cn[j] >= rem) {
        p.digit = 255 - 8 * lane - j;
        p.rem = rem - cum;
        p.whole = (rem - cum == cn[j]) ? 1 : 0;
        break;
      }
      cum += cn[j];
    }
  }
  p.digit = __shfl_sync(0xffffffffu, p.digit, src);
  p.rem = __shfl_sync(0xffffffffu, p.rem, src);
  p.whole = __shfl_sync(0xffffffffu, p.whole, src);
  return p;
}

__device__ __forceinline__ void cluster_arrive() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }

// Distributed shared memory pushes: the shared::cluster address of `a` (an
// address of this CTA's shared memory) in cluster CTA `rank`, and stores into
// a peer's shared memory that complete on the peer's mbarrier (transaction
// bytes), so the receiver needs no cluster-scope fence to read them.
__device__ __forceinline__ uint32_t peer_addr(uint32_t a, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
  return r;
}
__device__ __forceinline__ void push_v4(uint32_t dst, const int4& v, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.s32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(dst),
               "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(bar)
               : "memory");
}
__device__ __forceinline__ void push_v2(uint32_t dst, uint32_t x, uint32_t y, uint32_t bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.b32 [%0], {%1, %2}, [%3];" ::"r"(dst),
               "r"(x), "r"(y), "r"(bar)
               : "memory");
}

// Cluster radix select, grid (kTopnCluster, KV head, sequence), one cluster
// per (sequence, KV head). CTA r stages the order-preserving keys of blocks
// [r * per, (r + 1) * per) in shared memory. Every exchange between the CTAs
// is a push: a CTA stores its part (extremes, each pass's 256-bin histogram,
// its selected counts) into every CTA's receive buffer with stores that
// complete on the receiver's mbarrier, and each CTA waits on its own barrier
// for all eight parts. Only the barriers' initialisation needs a cluster
// barrier, whose arrive is issued at entry and whose wait comes before the
// first push. Each 8-bit pass builds a local histogram of the keys that still
// match the prefix; after the exchange every CTA sums the eight histograms
// and after one CTA barrier every warp finds the same digit (receive buffers
// alternate between passes: a CTA pushes pass p + 2 only after it received
// every CTA's pass p + 1, which each sent after reading its pass p buffer).
// The select stops early when the boundary bucket is taken whole. Then each
// CTA counts its keys above the boundary and at it; every warp reads the
// counts of the lower-ranked CTAs and of the lower warps and writes its
// selected ids in ascending order (ties at the boundary to the lower id).
// A wait that runs out records RESA_DEV_WAIT_TIMEOUT; the CTA then pushes
// nothing more and writes no ids. Every thread of every CTA arrives at one
// closing cluster barrier after its CTA's last push and waits on it just
// before it leaves, whether its waits succeeded or not.
// 40 registers (3 CTAs per SM): a CTA launched early then fits beside the
// persistent score CTA (88 registers x 512 threads), so its prologue runs
// before the scores are complete.
__global__ void __launch_bounds__(kTopnThreads, 3) topn_kernel(CacheView c, const float* __restrict__ scores,
                                                            double keep, int n_min, int n_local,
                                                            int32_t* __restrict__ indices,
                                                            int32_t* __restrict__ counts, int n_cap) {
  static_assert(kTopnThreads >= kTopnCluster * 32, "one 16-byte push per thread of the first 8 warps and pass");
  static_assert(kTopnSmemMax / sizeof(uint32_t) <= 0xFFFF, "a CTA's bin count fits 16 bits");
  extern __shared__ uint32_t keys[];
  __shared__ __align__(16) int hist[2][256];                     // local histogram of pass p in hist[p & 1]
  __shared__ __align__(16) uint16_t recv[2][kTopnCluster][256];  // every CTA's histogram of pass p in recv[p & 1]
  __shared__ __align__(16) int tot[256];
  __shared__ __align__(8) uint32_t recv_mm[kTopnCluster][2];  // every CTA's smallest and largest unforced key
  __shared__ __align__(8) int recv_cnt[kTopnCluster][2];      // every CTA's keys above / at the boundary
  __shared__ __align__(8) uint64_t bars[4];                   // passes (2, alternating), extremes, counts
  __shared__ int w_gt[kTopnWarps], w_eq[kTopnWarps];
  __shared__ uint32_t w_mm[kTopnWarps][2];
  uint32_t rank;
  asm("mov.u32 %0, %%cluster_ctarank;" : "=r"(rank));
  const int b = blockIdx.z, h = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t bar0 = smem_u32(&bars[0]);
  if (tid == 0) {
#pragma unroll
    for (int i = 0; i < 4; ++i) mbar_init(bar0 + 8 * i, 1);
    fence_mbar_init();
  }
  cluster_arrive();  // the barriers are initialised (waited for before the first push)
  for (int i = tid; i < 2 * 256; i += kTopnThreads) (&hist[0][0])[i] = 0;
  int32_t* out = indices + (static_cast<size_t>(b) * c.Hkv + h) * n_cap;
  const int T = __ldcg(c.seq_lens + b) + c.pending;  // final before the score kernel let this one launch
  pdl_wait();                                        // the scores
  pdl_launch_dependents();                           // after the wait: see the score kernel
  if (T < 0 || T > c.max_blocks * kBlock) {  // the whole cluster takes this branch
    if (rank == 0 && tid == 0) {
      record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
      counts[b * c.Hkv + h] = 0;
    }
    for (int i = static_cast<int>(rank) * kTopnThreads + tid; i < n_cap; i += kTopnCluster * kTopnThreads) out[i] = -1;
    cluster_wait();
    return;
  }
  const UnitBudget u = unit_budget(T, keep, n_min, n_local, n_cap, c.status, b * c.Hkv + h, rank == 0 && tid == 0);
  const int M = u.M, n = u.n, F = u.F, nf = u.nf, r = u.r;
  const int per = (M + kTopnCluster - 1) / kTopnCluster;
  const int lo = static_cast<int>(rank) * per, cnt = max(0, min(M, lo + per) - lo);
  const float* sc = scores + (static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks + lo;
  const int f_loc = F - lo;  // this CTA's ids >= f_loc are forced
  uint32_t kmin = 0xFFFFFFFFu, kmax = 0u;
  constexpr int kLoads = 8;  // loads in flight per thread
  for (int i0 = 0; i0 < cnt; i0 += kLoads * kTopnThreads) {
    float v[kLoads];
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
      const int i = i0 + k * kTopnThreads + tid;
      v[k] = i < cnt ? sc[i] : 0.f;
    }
#pragma unroll
    for (int k = 0; k < kLoads; ++k) {
      const int i = i0 + k * kTopnThreads + tid;
      if (i < cnt) {
        const uint32_t key = score_key(v[k]);
        keys[i] = key;
        if (i < f_loc) {
          kmin = min(kmin, key);
          kmax = max(kmax, key);
        }
      }
    }
  }
  // extreme unforced keys: per warp, per CTA (warp 0), then pushed to every CTA
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, o));
    kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
  }
  if (lane == 0) {
    w_mm[warp][0] = kmin;
    w_mm[warp][1] = kmax;
  }
  __syncthreads();  // the keys and every warp's extremes are visible
  cluster_wait();   // every CTA's barriers are initialised
  // `failed` (a wait ran out) is made uniform over the CTA at its barriers;
  // a CTA that failed pushes nothing more and skips its remaining waits.
  bool failed = false;
  if (warp == 0) {
    kmin = lane < kTopnWarps ? w_mm[lane][0] : 0xFFFFFFFFu;
    kmax = lane < kTopnWarps ? w_mm[lane][1] : 0u;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, o));
      kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
    }
    if (lane < kTopnCluster)
      push_v2(peer_addr(smem_u32(&recv_mm[rank][0]), lane), kmin, kmax, peer_addr(bar0 + 16, lane));
    if (lane == 0) mbar_arrive_expect_tx(bar0 + 16, kTopnCluster * 8);
  }
  failed |= !mbar_wait_bounded(bar0 + 16, 0);
  kmin = lane < kTopnCluster ? recv_mm[lane][0] : 0xFFFFFFFFu;
  kmax = lane < kTopnCluster ? recv_mm[lane][1] : 0u;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    kmin = min(kmin, __shfl_xor_sync(0xffffffffu, kmin, o));
    kmax = max(kmax, __shfl_xor_sync(0xffffffffu, kmax, o));
  }

  // ---- radix select of the r-th largest v = key - kmin among blocks [0, F) ----
  // The first digit is the top 8 significant bits of v, so the digits adapt
  // to the range of the unit's scores (which sit within a few per cent of
  // each other); r == 0 or r == F need no pass (prefix = pmask = 0).
  uint32_t prefix = 0, pmask = 0;
  int rem = r;
  if (r > 0 && r < F) {
    const int bits = 32 - __clz(static_cast<int>(kmax - kmin));  // significant bits of v
    int shift = max(bits - 8, 0), width = bits - shift;
    const int dst = tid >> 5, part = tid & 31;  // threads < 256: bins [8 part, 8 part + 8) to CTA dst
    for (int pass = 0;; ++pass) {
      const uint32_t dmask = (1u << width) - 1u;
      int* hb = hist[pass & 1];
      for (int i = tid; i < min(cnt, f_loc); i += kTopnThreads) {
        const uint32_t v = keys[i] - kmin;
        if ((v & pmask) == prefix) atomicAdd(&hb[(v >> shift) & dmask], 1);
      }
      failed = __syncthreads_or(failed);  // this CTA's histogram of the pass is complete
      if (!failed) {
        const uint32_t bar = bar0 + 8 * (pass & 1);
        if (tid < kTopnCluster * 32) {
          const int4 a = reinterpret_cast<const int4*>(hb)[2 * part], e = reinterpret_cast<const int4*>(hb)[2 * part + 1];
          const int4 v = make_int4(a.x | (a.y << 16), a.z | (a.w << 16), e.x | (e.y << 16), e.z | (e.w << 16));
          push_v4(peer_addr(smem_u32(&recv[pass & 1][rank][8 * part]), dst), v, peer_addr(bar, dst));
        }
        if (tid == 0) mbar_arrive_expect_tx(bar, kTopnCluster * 256 * sizeof(uint16_t));
        failed = !mbar_wait_bounded(bar, (pass >> 1) & 1);
      }
      if (tid < 256) {
        int t = 0;
#pragma unroll
        for (int q = 0; q < kTopnCluster; ++q) t += recv[pass & 1][q][tid];
        tot[tid] = t;
      }
      failed = __syncthreads_or(failed);  // the cluster's histogram is visible; every thread has pushed this pass
      for (int i = tid; i < 256; i += kTopnThreads) hb[i] = 0;  // for pass + 2 (the next barrier orders it)
      const DigitPick pk = pick_digit(tot, rem);  // the same in every warp and every CTA
      prefix |= static_cast<uint32_t>(pk.digit) << shift;
      pmask |= dmask << shift;
      rem = pk.rem;
      if (pk.whole || shift == 0) break;
      width = min(8, shift);
      shift -= width;
    }
  }
  // Selected: forced blocks [F, F + nf), and among [0, F) the ids with
  // (v & pmask) > prefix, or == prefix among the first `take_eq` such ids in
  // block order.
  const int take_eq = rem;
  auto classify = [&](int i, bool in, bool& is_gt, bool& is_eq) {  // local id i
    is_gt = false;
    is_eq = false;
    if (in) {
      if (i >= f_loc) {
        is_gt = lo + i - F < nf;
      } else {
        const uint32_t v = (keys[i] - kmin) & pmask;
        is_gt = v > prefix;
        is_eq = v == prefix;
      }
    }
  };

  // ---- ordered compaction: warps own contiguous id ranges of the CTA ----
  const int per_warp = ((cnt + 31) / 32 + kTopnWarps - 1) / kTopnWarps * 32;
  const int w0 = warp * per_warp, w1 = min(cnt, w0 + per_warp);
  int gt = 0, eq = 0;
  for (int i0 = w0; i0 < w1; i0 += 32) {
    bool is_gt, is_eq;
    classify(i0 + lane, i0 + lane < w1, is_gt, is_eq);
    gt += __popc(__ballot_sync(0xffffffffu, is_gt));
    eq += __popc(__ballot_sync(0xffffffffu, is_eq));
  }
  if (lane == 0) {
    w_gt[warp] = gt;
    w_eq[warp] = eq;
  }
  failed = __syncthreads_or(failed);
  // this CTA's totals (every warp computes them; warp 0 pushes them to every CTA)
  const int g_l = lane < kTopnWarps ? w_gt[lane] : 0, e_l = lane < kTopnWarps ? w_eq[lane] : 0;
  const int g_in = warp_incl_scan(g_l), e_in = warp_incl_scan(e_l);
  if (!failed) {
    if (warp == 0) {
      const int gt_cta = __shfl_sync(0xffffffffu, g_in, 31), eq_cta = __shfl_sync(0xffffffffu, e_in, 31);
      if (lane < kTopnCluster)
        push_v2(peer_addr(smem_u32(&recv_cnt[rank][0]), lane), static_cast<uint32_t>(gt_cta),
                static_cast<uint32_t>(eq_cta), peer_addr(bar0 + 24, lane));
      if (lane == 0) mbar_arrive_expect_tx(bar0 + 24, kTopnCluster * 8);
    }
    failed = __any_sync(0xffffffffu, !mbar_wait_bounded(bar0 + 24, 0));
  }
  // lower-ranked CTAs: lane q < rank reads CTA q's counts
  int gq = 0, eqq = 0;
  if (lane < static_cast<int>(rank)) {
    gq = recv_cnt[lane][0];
    eqq = recv_cnt[lane][1];
  }
  const int eq_incl = warp_incl_scan(eqq);
  const int sel_q = gq + max(0, min(eqq, take_eq - (eq_incl - eqq)));
  int sel_before = sel_q;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) sel_before += __shfl_xor_sync(0xffffffffu, sel_before, o);
  const int eq_before = __shfl_sync(0xffffffffu, eq_incl, 31);
  // lower warps of this CTA
  const int e_ex = e_in - e_l;
  const int s_l = g_l + max(0, min(e_l, take_eq - (eq_before + e_ex)));
  const int s_in = warp_incl_scan(s_l);
  int eq_seen = eq_before + __shfl_sync(0xffffffffu, e_ex, warp);
  int pos = sel_before + __shfl_sync(0xffffffffu, s_in - s_l, warp);
  // Closing cluster barrier, split: every thread arrives here, after its
  // CTA's last push, and waits just before it leaves, on the success and the
  // failure path alike, so no CTA leaves while a peer may still push into its
  // shared memory (a CTA that timed out stops pushing, but its peers may not
  // have noticed yet).
  asm volatile("barrier.cluster.arrive.release;" ::: "memory");
  if (failed) {  // (warp-uniform) values received may be incomplete: write no ids
    if (lane == 0) record_error(c.status, RESA_DEV_WAIT_TIMEOUT, b * c.Hkv + h);
    asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
    return;
  }
  for (int i0 = w0; i0 < w1; i0 += 32) {
    const int i = i0 + lane;
    bool is_gt, is_eq;
    classify(i, i < w1, is_gt, is_eq);
    const unsigned eqm = __ballot_sync(0xffffffffu, is_eq);
    const int my_eq_rank = eq_seen + __popc(eqm & ((1u << lane) - 1u));
    const bool sel = is_gt || (is_eq && my_eq_rank < take_eq);
    const unsigned selm = __ballot_sync(0xffffffffu, sel);
    if (sel) out[pos + __popc(selm & ((1u << lane) - 1u))] = lo + i;
    eq_seen += __popc(eqm);
    pos += __popc(selm);
  }
  for (int i = n + static_cast<int>(rank) * kTopnThreads + tid; i < n_cap; i += kTopnCluster * kTopnThreads) out[i] = -1;
  if (rank == 0 && tid == 0) counts[b * c.Hkv + h] = n;
  asm volatile("barrier.cluster.wait.acquire;" ::: "memory");
}

// One-CTA radix select, grid (KV head, sequence), for caches of up to
// kTopnCtaMaxBlocks blocks per sequence: the same selection as topn_kernel
// with every barrier a CTA barrier. Warp w owns the contiguous id range
// [w * per_warp, (w + 1) * per_warp) and its lane l the ids w * per_warp +
// 32 j + l, whose keys it keeps in registers from staging to compaction: a
// pass reads no shared memory but the histogram, and its shared-memory
// atomics are independent of one another. The histograms rotate through
// three buffers, so one barrier per pass suffices (the buffer zeroed during a
// pass was last read two passes before); warp 0 finds each digit and one
// more barrier hands it to the other warps. Every warp derives its output
// offset from the per-warp counts after a single barrier.
template <int kKeys>
__global__ void __launch_bounds__(kTopnCtaThreads, 2) topn_cta_kernel(CacheView c, const float* __restrict__ scores,
                                                                      double keep, int n_min, int n_local,
                                                                      int32_t* __restrict__ indices,
                                                                      int32_t* __restrict__ counts, int n_cap) {
  __shared__ __align__(16) int hist[3][256];
  __shared__ uint32_t w_lo[kTopnCtaWarps], w_hi[kTopnCtaWarps];
  __shared__ int w_gt[kTopnCtaWarps], w_eq[kTopnCtaWarps];
  __shared__ int sh_pick[3];  // digit, rank left, whole bucket taken
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < 2 * 256; i += kTopnCtaThreads) (&hist[0][0])[i] = 0;
  const int h = blockIdx.x, b = blockIdx.y;
  int32_t* out = indices + (static_cast<size_t>(b) * c.Hkv + h) * n_cap;
  const int T = __ldcg(c.seq_lens + b) + c.pending;  // final before the score kernel let this one launch
  if (T < 0 || T > c.max_blocks * kBlock) {
    pdl_wait();
    pdl_launch_dependents();
    if (tid == 0) {
      record_error(c.status, RESA_DEV_SEQ_LEN_RANGE, b);
      counts[b * c.Hkv + h] = 0;
    }
    for (int i = tid; i < n_cap; i += kTopnCtaThreads) out[i] = -1;
    return;
  }
  const UnitBudget u = unit_budget(T, keep, n_min, n_local, n_cap, c.status, b * c.Hkv + h, tid == 0);
  const int M = u.M, n = u.n, F = u.F, nf = u.nf, r = u.r;
  const int per_warp = ((M + 31) / 32 + kTopnCtaWarps - 1) / kTopnCtaWarps * 32;  // <= 32 kKeys (the launch picks kKeys)
  const int w0 = warp * per_warp;
  // bit j: id w0 + 32 j + lane is a candidate (< F) / a forced block taken ([F, F + nf))
  uint32_t cand = 0, forced = 0;
#pragma unroll
  for (int j = 0; j < kKeys; ++j) {
    const int i = w0 + 32 * j + lane;
    if (32 * j < per_warp) {
      if (i < F) cand |= 1u << j;
      else if (i - F < nf) forced |= 1u << j;
    }
  }
  const float* sc = scores + (static_cast<size_t>(b) * c.Hkv + h) * c.max_blocks + w0 + lane;
  pdl_wait();  // the scores
  pdl_launch_dependents();  // after the wait: see the score kernel
  uint32_t key[kKeys];
#pragma unroll
  for (int j = 0; j < kKeys; ++j) key[j] = (cand >> j) & 1u ? score_key(sc[32 * j]) : 0u;
  uint32_t kmin = 0xFFFFFFFFu, kmax = 0u;
#pragma unroll
  for (int j = 0; j < kKeys; ++j)
    if ((cand >> j) & 1u) {
      kmin = min(kmin, key[j]);
      kmax = max(kmax, key[j]);
    }
  kmin = __reduce_min_sync(0xffffffffu, kmin);
  kmax = __reduce_max_sync(0xffffffffu, kmax);
  if (lane == 0) {
    w_lo[warp] = kmin;
    w_hi[warp] = kmax;
  }
  __syncthreads();  // the per-warp extremes are visible
  kmin = __reduce_min_sync(0xffffffffu, lane < kTopnCtaWarps ? w_lo[lane] : 0xFFFFFFFFu);
  kmax = __reduce_max_sync(0xffffffffu, lane < kTopnCtaWarps ? w_hi[lane] : 0u);
#pragma unroll
  for (int j = 0; j < kKeys; ++j) key[j] -= kmin;  // v = key - min key (candidates only are read)

  // ---- radix select of the r-th largest v among blocks [0, F) ----
  uint32_t prefix = 0, pmask = 0;
  int rem = r;
  if (r > 0 && r < F) {
    const int bits = 32 - __clz(static_cast<int>(kmax - kmin));  // significant bits of v
    int shift = max(bits - 8, 0), width = bits - shift;
    for (int pass = 0;; ++pass) {
      const uint32_t dmask = (1u << width) - 1u;
      int* hb = hist[pass % 3];
      if (tid < 256) hist[(pass + 1) % 3][tid] = 0;
#pragma unroll
      for (int j = 0; j < kKeys; ++j)
        if (((cand >> j) & 1u) && (key[j] & pmask) == prefix) atomicAdd(&hb[(key[j] >> shift) & dmask], 1);
      __syncthreads();  // this pass's histogram is complete
      if (warp == 0) {
        const DigitPick pk = pick_digit(hb, rem);
        if (lane == 0) {
          sh_pick[0] = pk.digit;
          sh_pick[1] = pk.rem;
          sh_pick[2] = pk.whole;
        }
      }
      __syncthreads();  // the digit is visible
      prefix |= static_cast<uint32_t>(sh_pick[0]) << shift;
      pmask |= dmask << shift;
      rem = sh_pick[1];
      if (sh_pick[2] || shift == 0) break;
      width = min(8, shift);
      shift -= width;
    }
  }
  // Selected: the forced blocks, and among the candidates the ids with
  // (v & pmask) > prefix, or == prefix among the first `take_eq` such ids.
  const int take_eq = rem;
  uint32_t gtm = forced, eqm = 0;
#pragma unroll
  for (int j = 0; j < kKeys; ++j)
    if ((cand >> j) & 1u) {
      const uint32_t v = key[j] & pmask;
      if (v > prefix) gtm |= 1u << j;
      else if (v == prefix) eqm |= 1u << j;
    }
  const int gt = __reduce_add_sync(0xffffffffu, __popc(gtm)), eq = __reduce_add_sync(0xffffffffu, __popc(eqm));
  if (lane == 0) {
    w_gt[warp] = gt;
    w_eq[warp] = eq;
  }
  __syncthreads();  // every warp's counts are visible
  // this warp's offsets: equal keys and selected ids of the lower warps
  const int e_l = lane < kTopnCtaWarps ? w_eq[lane] : 0, g_l = lane < kTopnCtaWarps ? w_gt[lane] : 0;
  const int ie = warp_incl_scan(e_l);
  const int s_l = g_l + max(0, min(e_l, take_eq - (ie - e_l)));
  const int is = warp_incl_scan(s_l);
  int eq_seen = __shfl_sync(0xffffffffu, ie - e_l, warp);
  int pos = __shfl_sync(0xffffffffu, is - s_l, warp);
  const unsigned below = (1u << lane) - 1u;
#pragma unroll
  for (int j = 0; j < kKeys; ++j) {
    if (32 * j >= per_warp) break;
    const bool is_eq = (eqm >> j) & 1u;
    const unsigned eqb = __ballot_sync(0xffffffffu, is_eq);
    const bool sel = ((gtm >> j) & 1u) || (is_eq && eq_seen + __popc(eqb & below) < take_eq);
    const unsigned selb = __ballot_sync(0xffffffffu, sel);
    if (sel) out[pos + __popc(selb & below)] = w0 + 32 * j + lane;
    eq_seen += __popc(eqb);
    pos += __popc(selb);
  }
  for (int i = n + tid; i < n_cap; i += kTopnCtaThreads) out[i] = -1;
  if (tid == 0) counts[b * c.Hkv + h] = n;
}

}  // namespace

size_t select_smem_bytes(int max_blocks) {
  if (max_blocks <= kTopnCtaMaxBlocks) return 0;  // keys in registers
  return static_cast<size_t>((max_blocks + kTopnCluster - 1) / kTopnCluster) * sizeof(uint32_t);
}

int select_max_blocks() { return kTopnCluster * (kTopnSmemMax / static_cast<int>(sizeof(uint32_t))); }

template <int kPieceBlocks, int kScoreStages>
cudaError_t launch_score(const CacheView& c, const uint16_t* q, float* scores, int sm_count, cudaStream_t st,
                         int attr_slot) {
  constexpr int kSmem = score_smem_bytes(kPieceBlocks, kScoreStages);
  const auto kernel = score_kernel<kPieceBlocks, kScoreStages>;
  cudaError_t e =
      ensure_smem_attr(reinterpret_cast<const void*>(kernel), kSmem + score_table_bytes(kMaxBatch), attr_slot);
  if (e != cudaSuccess) return e;
  // one persistent CTA per SM (never more than the pieces there can be)
  const long long max_pieces =
      static_cast<long long>(c.B) * c.Hkv * ((c.max_blocks + kPieceBlocks - 1) / kPieceBlocks);
  const int grid = static_cast<int>(max(1LL, min(static_cast<long long>(sm_count), max_pieces)));
  return launch_pdl(kernel, dim3(grid), dim3(kScoreWarps * 32), kSmem + score_table_bytes(c.B), st, c, q, scores);
}

cudaError_t launch_select(const CacheView& c, const uint16_t* q, double keep, int n_min, int n_local,
                          int32_t* indices, int32_t* counts, int n_cap, float* scores, int sm_count,
                          cudaStream_t st) {
  // 6 KB pieces when there is at least one per warp of a full grid
  const long long pieces12 = static_cast<long long>(c.B) * c.Hkv * ((c.max_blocks + 11) / 12);
  cudaError_t e = pieces12 >= static_cast<long long>(sm_count) * kScoreWarps
                      ? launch_score<12, 2>(c, q, scores, sm_count, st, 3)
                      : launch_score<8, 3>(c, q, scores, sm_count, st, 4);
  if (e != cudaSuccess) return e;
  const size_t smem = select_smem_bytes(c.max_blocks);
  if (c.max_blocks <= kTopnCtaMaxBlocks) {
    // key slots per thread for the cache's largest unit: the loops over the
    // slots unroll to the smallest instantiation that holds them
    const int slots = ((c.max_blocks + 31) / 32 + kTopnCtaWarps - 1) / kTopnCtaWarps;
    const auto kernel = slots <= 1   ? topn_cta_kernel<1>
                        : slots <= 2 ? topn_cta_kernel<2>
                        : slots <= 3 ? topn_cta_kernel<3>
                        : slots <= 4 ? topn_cta_kernel<4>
                        : slots <= 5 ? topn_cta_kernel<5>
                        : slots <= 6 ? topn_cta_kernel<6>
                        : slots <= 8 ? topn_cta_kernel<8>
                                     : topn_cta_kernel<kTopnCtaKeys>;
    return launch_pdl(kernel, dim3(c.Hkv, c.B), dim3(kTopnCtaThreads), smem, st, c,
                      static_cast<const float*>(scores), keep, n_min, n_local, indices, counts, n_cap);
  }
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
