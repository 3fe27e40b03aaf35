/*
 * resa.h -- C ABI of the GB300 (sm_103a) decode-time attention path of
 * Rectified Sparse Attention (ReSA, arXiv 2506.04108).
 *
 * The path, per decode step of a batch of sequences:
 *   resa_commit_kv(append)      Algorithm 1: update the KV cache and block-key
 *                               cache with the new token (Eq. 3, online).
 *   resa_select_blocks          Eq. 4 + Eq. 5: pooled GQA-group query, Quest
 *                               block scores, dynamic top-n with forced local
 *                               blocks; one block set per KV head.
 *   resa_sparse_decode          Eq. 2 / Algorithm 2: split-K flash decoding
 *                               over the selected blocks, then the combine.
 * and every f steps (Algorithm 1, rectification branch):
 *   resa_rectify_attention      dense causal attention of the last f tokens
 *                               against the whole cache (Section 2.2).
 *   resa_commit_kv(overwrite)   write back their dense K/V and recompute the
 *                               touched block summaries.
 *   resa_update_summaries       Eq. 3 over a range of blocks (prefill / bulk).
 *
 * Conventions shared by every call
 *   - All tensor pointers are DEVICE pointers owned by the caller; the library
 *     never allocates, frees, synchronises (except resa_read_device_error) or
 *     aborts. Every compute call is asynchronous on `stream` (a cudaStream_t
 *     passed as void*; NULL is the legacy default stream).
 *   - bf16 is IEEE bfloat16 (uint16 storage); accumulation is fp32.
 *   - Arguments are validated on the host before any launch; a bad argument
 *     returns an error code and launches nothing.
 *   - Conditions only the device can see (a sequence length out of range, a
 *     page id out of range, a budget above n_cap, a bounded wait that ran
 *     out) are recorded in cache->device_status (first error wins) and the
 *     affected work is skipped; resa_read_device_error() returns them.
 *   - Supported geometry: head_dim 128, block_size 16, GQA group size
 *     num_q_heads / num_kv_heads in [1, 8], batch <= 1024, and
 *     max_blocks_per_seq <= 409600 (6.5M tokens); other values return
 *     RESA_ERR_UNSUPPORTED.
 *   - The library is stateless apart from per-device cached attributes and is
 *     safe to call from several host threads; calls that share buffers must
 *     be ordered by the caller (same stream or events).
 */
#ifndef RESA_H_
#define RESA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RESA_ABI_VERSION 1

typedef enum resa_status {
  RESA_OK = 0,
  RESA_ERR_INVALID_ARG = 1,   /* null pointer, negative size, inconsistent shape */
  RESA_ERR_UNSUPPORTED = 2,   /* head_dim != 128, block_size != 16, group > 8, ... */
  RESA_ERR_WORKSPACE = 3,     /* workspace missing or smaller than required */
  RESA_ERR_CUDA = 4,          /* a CUDA runtime call failed (launch, attribute) */
  RESA_ERR_DEVICE = 5         /* resa_read_device_error found a device-side error */
} resa_status_t;

/* Codes written to device_status[0] by kernels (device_status[1] = detail). */
typedef enum resa_device_error {
  RESA_DEV_OK = 0,
  RESA_DEV_SEQ_LEN_RANGE = 1,    /* seq_lens[b] < 0, > capacity, or too short for the call */
  RESA_DEV_PAGE_RANGE = 2,       /* page_table entry outside [0, num_pages) */
  RESA_DEV_BUDGET_OVER_CAP = 3,  /* selection budget n exceeded n_cap (clamped to n_cap) */
  RESA_DEV_WAIT_TIMEOUT = 4,     /* a bounded barrier wait ran out (work skipped) */
  RESA_DEV_BAD_INDEX = 5         /* a block index / count passed to decode is out of range */
} resa_device_error_t;

/*
 * The paged KV cache (Algorithm 1's K) and block-key cache (B).
 *
 *   k_pool, v_pool  bf16 [num_pages][num_kv_heads][block_size][head_dim].
 *                   One page holds one block of block_size consecutive tokens
 *                   of one sequence for all KV heads; block i of sequence b
 *                   lives in page page_table[b][i] (the blocks of Eq. 2/3).
 *   page_table      int32 [batch][max_blocks_per_seq], logical block -> page.
 *   seq_lens        int32 [batch], tokens currently in each sequence (T).
 *                   Device resident so that a captured CUDA graph replays
 *                   correctly as sequences grow; resa_commit_kv(append)
 *                   advances it.
 *   summaries       bf16 [batch][num_kv_heads][max_blocks_per_seq][2][head_dim]:
 *                   element-wise min ([..][0][..]) and max ([..][1][..]) of
 *                   the valid keys of each block (Eq. 3).
 *   device_status   int32 [4], zero-initialised by the caller; kernels record
 *                   the first device-side error here.
 * Capacity of a sequence is max_blocks_per_seq * block_size tokens.
 */
typedef struct resa_cache {
  int32_t batch;
  int32_t num_q_heads;
  int32_t num_kv_heads;
  int32_t head_dim;
  int32_t block_size;
  int32_t num_pages;
  int32_t max_blocks_per_seq;
  int32_t reserved0;
  void* k_pool;
  void* v_pool;
  const int32_t* page_table;
  int32_t* seq_lens;
  void* summaries;
  int32_t* device_status;
} resa_cache_t;

/*
 * ReSA selection and attention parameters (Section 2.1, Eq. 5; Section 3.1).
 *   keep_ratio      fraction of blocks attended: n = max(n_min_blocks,
 *                   ceil(M * keep_ratio)) evaluated on the float64 product,
 *                   M = ceil(T / block_size). The paper's "sparsity 0.9" is
 *                   keep_ratio 0.1. In [0, 1].
 *   n_min_blocks    minimum budget n_min (>= 0).
 *   n_local_blocks  the n_local most recent blocks are always selected (their
 *                   score is set to +inf); they count inside n, and
 *                   n >= n_local_blocks, n <= M.
 *   sm_scale        softmax scale of q.k; 0 selects 1/sqrt(head_dim).
 */
typedef struct resa_params {
  double keep_ratio;
  int32_t n_min_blocks;
  int32_t n_local_blocks;
  float sm_scale;
  int32_t reserved0;
} resa_params_t;

/* ABI version of the loaded library (RESA_ABI_VERSION at build time). */
int32_t resa_abi_version(void);

/* Human-readable name of a status code (static storage, never NULL). */
const char* resa_status_string(resa_status_t status);

/*
 * Largest selection budget any sequence of this cache can reach: the n of
 * Eq. 5 at M = max_blocks_per_seq. Passing n_cap >= this value to
 * resa_select_blocks guarantees RESA_DEV_BUDGET_OVER_CAP never fires.
 */
resa_status_t resa_max_selected(const resa_cache_t* cache, const resa_params_t* params, int32_t* n_out);

/*
 * Number of key splits resa_sparse_decode uses when num_splits == 0, for the
 * current device: Algorithm 2's num_splits, chosen so that
 * batch * num_kv_heads * splits fills the SMs in one wave (Section 2.4), with
 * one resident CTA per SM instead of two when two would leave a split fewer
 * than 16 of the n_cap selected blocks, and at least two blocks per split.
 */
resa_status_t resa_decode_num_splits(const resa_cache_t* cache, int32_t n_cap, int32_t* splits_out);

/*
 * Number of key splits resa_rectify_attention uses for f new tokens on the
 * current device (Section 2.2; the dense pass is split over the cached keys
 * like Algorithm 2 splits the decode): the query rows of a KV head form
 * ceil(8 f / 256) row groups of up to 256 rows (token-major, heads padded to
 * 8), and splits = SMs / (batch * num_kv_heads * row groups), at least 1 and
 * at most the 64-key tiles of the cache's capacity and 256. Split s of a
 * sequence with T tokens takes the 64-key tiles [s * per, (s + 1) * per) of
 * its prefix [0, T - f), per = ceil(ceil((T - f) / 64) / splits); the last
 * split also takes the f new tokens.
 */
resa_status_t resa_rectify_num_splits(const resa_cache_t* cache, int32_t f, int32_t* splits_out);

/*
 * Bytes of scratch workspace the compute calls need for this cache:
 * resa_select_blocks (block scores), resa_sparse_decode with `num_splits`
 * (0 = auto) at budget cap n_cap (split partials), and
 * resa_rectify_attention with f <= max_f (key-split partials). One buffer of
 * this size may be shared by all calls issued in order on one stream.
 * Requires a current CUDA device (the SM count sizes the splits).
 */
resa_status_t resa_workspace_size(const resa_cache_t* cache, int32_t n_cap, int32_t num_splits, int32_t max_f,
                                  size_t* bytes_out);

/*
 * Eq. 3 over a range of blocks: for every sequence b and KV head, recompute
 * summaries[b][h][i] for blocks i in [block_begin, block_end) that hold at
 * least one valid token (i * block_size < seq_lens[b]); block_end = -1 means
 * "through the last block of each sequence". Blocks are recomputed from the
 * cached keys of positions < seq_lens[b] (a partial last block covers only
 * its valid tokens). Used after a prefill and for bulk refreshes.
 */
resa_status_t resa_update_summaries(const resa_cache_t* cache, int32_t block_begin, int32_t block_end,
                                    void* stream);

/*
 * Algorithm 1, "update KV cache / block key cache":
 *   k_new, v_new  bf16 [batch][n_tokens][num_kv_heads][head_dim].
 *   overwrite = 0 (append):    token t is written at position seq_lens[b] + t,
 *                              the summaries of the touched blocks are updated
 *                              online (min/max with the new keys; exact), then
 *                              seq_lens[b] += n_tokens.
 *   overwrite = 1 (rectify):   token t is written at position
 *                              seq_lens[b] - n_tokens + t (the rectification
 *                              write-back of Section 2.2); every touched block
 *                              is recomputed from all its valid keys;
 *                              seq_lens is unchanged.
 * Device errors: a write beyond capacity or before position 0 skips the
 * sequence and records RESA_DEV_SEQ_LEN_RANGE.
 */
resa_status_t resa_commit_kv(const resa_cache_t* cache, const void* k_new, const void* v_new, int32_t n_tokens,
                             int32_t overwrite, void* stream);

/*
 * Eq. 4 + Eq. 5 (Section 2.1, "Block Selection"), one block set per
 * (sequence, KV head), shared by the group's query heads:
 *   q         bf16 [batch][num_q_heads][head_dim]; query head j belongs to KV
 *             head j / (num_q_heads / num_kv_heads).
 *   The pooled query is the mean of the group's query heads (fp32); block i's
 *   score is sum_j max(q_j * kmax_ij, q_j * kmin_ij) over the summaries, for
 *   i < M = ceil(seq_lens[b] / block_size); the last n_local blocks score
 *   +inf; the n highest scores are kept, ties to the lower block index.
 *   indices   int32 [batch][num_kv_heads][n_cap]: selected block ids in
 *             ascending order, then -1 padding.
 *   counts    int32 [batch][num_kv_heads]: n for each row.
 * Workspace: at least resa_workspace_size(); holds fp32 scores.
 */
resa_status_t resa_select_blocks(const resa_cache_t* cache, const void* q, const resa_params_t* params,
                                 int32_t* indices, int32_t* counts, int32_t n_cap, void* workspace,
                                 size_t workspace_bytes, void* stream);

/*
 * Eq. 2 (GBSA) computed as Algorithm 2: grid (splits, num_kv_heads, batch);
 * each CTA loads the group's queries, attends to its share of the selected
 * blocks (keys at positions >= seq_lens[b] are masked), and stores a partial
 * output and log-sum-exp; a combine kernel merges the splits.
 *   q         bf16 [batch][num_q_heads][head_dim]
 *   indices, counts, n_cap   as produced by resa_select_blocks (any ascending
 *             or unordered set of distinct in-range block ids is accepted).
 *   out       bf16 [batch][num_q_heads][head_dim]
 *   lse       fp32 [batch][num_q_heads] or NULL: natural log of the softmax
 *             denominator of the scaled logits (-inf if nothing attended).
 *   num_splits  Algorithm 2's num_splits; 0 = resa_decode_num_splits().
 */
resa_status_t resa_sparse_decode(const resa_cache_t* cache, const void* q, const int32_t* indices,
                                 const int32_t* counts, int32_t n_cap, const resa_params_t* params, void* out,
                                 float* lse, int32_t num_splits, void* workspace, size_t workspace_bytes,
                                 void* stream);

/*
 * One sparse decode step of Algorithm 1 in one call: the append commit of one
 * token (k_new, v_new; bf16 [batch][num_kv_heads][head_dim]), block
 * selection (Eq. 4, Eq. 5) and block-sparse decoding (Eq. 2, Algorithm 2) --
 * the same results, bit for bit, as resa_commit_kv(n_tokens = 1, append)
 * followed by resa_select_blocks and resa_sparse_decode on the same arguments,
 * without the commit's own launch: the scoring pass writes the new key and
 * value into their page and folds the key into its block's summary before it
 * scores that block, and the combine kernel advances seq_lens[b] by one at the
 * end. Arguments are those of the three calls; the workspace must hold both
 * the scores and the split partials (resa_workspace_size covers it).
 * Device errors: as in the three calls; a sequence already at capacity is
 * reported (RESA_DEV_SEQ_LEN_RANGE), gets count 0, and keeps its length.
 */
resa_status_t resa_decode_step(const resa_cache_t* cache, const void* k_new, const void* v_new, const void* q,
                               const resa_params_t* params, int32_t* indices, int32_t* counts, int32_t n_cap,
                               void* out, float* lse, int32_t num_splits, void* workspace, size_t workspace_bytes,
                               void* stream);

/*
 * Dense rectification attention (Section 2.2; Algorithm 1 DenseForward):
 * the f most recent tokens of each sequence, at positions
 * [seq_lens[b] - f, seq_lens[b]), attend causally to the whole cache: query
 * row i sees positions [0, seq_lens[b] - f + i]. Keys/values of positions
 * < seq_lens[b] - f come from the cache; those of the f tokens come from
 * k_new / v_new (the dense re-encode), so calling this before or after the
 * overwrite commit gives the same result.
 *   q_new     bf16 [batch][f][num_q_heads][head_dim]
 *   k_new, v_new  bf16 [batch][f][num_kv_heads][head_dim]
 *   out       bf16 [batch][f][num_q_heads][head_dim]
 *   lse       fp32 [batch][f][num_q_heads] or NULL (natural log).
 * Device errors: seq_lens[b] < f records RESA_DEV_SEQ_LEN_RANGE.
 * The same call is the attention of Algorithm 1's dense prefill done in
 * chunks: after resa_commit_kv(append) of a chunk of C prompt tokens (which
 * also builds their block keys), f = C attends the chunk's queries causally
 * to the cached prefix and to the chunk itself.
 */
resa_status_t resa_rectify_attention(const resa_cache_t* cache, const void* q_new, const void* k_new,
                                     const void* v_new, int32_t f, const resa_params_t* params, void* out,
                                     float* lse, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Continuous batching (requests at different points of their own rectification
 * period share a batch): resa_commit_kv and resa_rectify_attention restricted
 * to the sequences b with active[b] != 0. The others are left exactly as they
 * are: no cache, length or summary change, no output row written, no device
 * error recorded for them. active: int32 [batch] on the device (NULL = all,
 * which is what the plain calls do). Everything else is as in the plain calls.
 */
resa_status_t resa_commit_kv_active(const resa_cache_t* cache, const int32_t* active, const void* k_new,
                                    const void* v_new, int32_t n_tokens, int32_t overwrite, void* stream);
resa_status_t resa_rectify_attention_active(const resa_cache_t* cache, const int32_t* active, const void* q_new,
                                            const void* k_new, const void* v_new, int32_t f,
                                            const resa_params_t* params, void* out, float* lse, void* workspace,
                                            size_t workspace_bytes, void* stream);

/*
 * resa_sparse_decode without a caller workspace. The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory --
 * for example a plugin inside a host framework that owns all device memory
 * and hands its plugins no allocator, or code on a latency-critical path
 * where a device allocation (which may synchronise the device) is not
 * allowed. It computes exactly what resa_sparse_decode computes, with the
 * same arguments minus the workspace; the split partials live instead in one
 * library-owned static device buffer of RESA_STATIC_SCRATCH_BYTES, which
 * every GPU that loads the library holds until the process exits.
 *   - It calls no cudaMalloc / cudaFree or any allocating routine.
 *   - Calls whose partials need more than RESA_STATIC_SCRATCH_BYTES
 *     (batch * num_q_heads * splits * (head_dim + 1) * 4 bytes, each part
 *     rounded up to 256 bytes) return RESA_ERR_WORKSPACE and launch nothing.
 *   - The first call on a device looks up the buffer's device address (with
 *     that device current) and caches it for the rest of the process; make
 *     that first call before any stream capture on that device. The cached
 *     address belongs to the device's primary context: after cudaDeviceReset
 *     (or anything else that destroys that context) it is stale, and this
 *     entry point must not be called again in that process.
 *   - All calls share the one buffer, and it keeps the last call's contents
 *     (nothing in it needs to start at zero: every call overwrites every
 *     partial it reads). Calls that overlap on the GPU (e.g. on two streams
 *     without ordering) race on the buffer and give undefined results.
 */
#define RESA_STATIC_SCRATCH_BYTES (4u * 1024u * 1024u)
resa_status_t resa_sparse_decode_static(const resa_cache_t* cache, const void* q, const int32_t* indices,
                                        const int32_t* counts, int32_t n_cap, const resa_params_t* params,
                                        void* out, float* lse, int32_t num_splits, void* stream);

/*
 * Failure-detection hook of the sparse decode kernel (resa_sparse_decode,
 * resa_decode_step, resa_sparse_decode_static). Each warp of that kernel
 * waits for the copies of its K/V blocks on shared-memory barriers, and
 * gives up after `polls` polls of one barrier phase: it then records
 * RESA_DEV_WAIT_TIMEOUT in device_status, skips its remaining blocks (the
 * partial output covers the blocks attended before the wait ran out; a warp
 * that attended none contributes nothing, so an output row whose every warp
 * gave up is zero with lse -inf), and still waits, with the default limit,
 * for every copy it had issued before its CTA exits, so no copy lands in
 * released shared memory. The default, RESA_DEFAULT_DECODE_WAIT_POLLS, only
 * runs out if a copy never completes; 0 makes every wait give up at once,
 * which lets a test drive the timeout path without a fault or a hang. The
 * setting is process-wide and read when a call is issued (a captured graph
 * keeps the value of its capture). Always returns RESA_OK.
 */
#define RESA_DEFAULT_DECODE_WAIT_POLLS (1u << 22)
resa_status_t resa_set_decode_wait_polls(uint32_t polls);

/*
 * Synchronises `stream`, then copies device_status[0..1] to *code_out /
 * *detail_out (either may be NULL) and clears device_status. Returns
 * RESA_ERR_DEVICE if a device error had been recorded, RESA_OK otherwise.
 */
resa_status_t resa_read_device_error(const resa_cache_t* cache, int32_t* code_out, int32_t* detail_out,
                                     void* stream);

#ifdef __cplusplus
}
#endif

#endif /* RESA_H_ */
