"""fp64 CPU oracle of the ReSA decode-time attention path.

TEST INFRASTRUCTURE ONLY. Nothing in the product path may import or call
this module: only the tests, the smoke check and the benchmark's CPU-baseline
leg do. It shares no code with the CUDA library.

Plain, slow, obviously correct numpy in float64. bf16 inputs are widened
exactly to float64 before any arithmetic. Each function names the part of the
paper (arXiv 2506.04108) it follows:

* Eq. 1  GQA attention, softmax(q K^T / sqrt(d)) V.
* Eq. 2  group block-sparse attention (GBSA): only keys of selected blocks.
* Eq. 3  per-block element-wise key min / max.
* Eq. 4  Quest block score of the pooled group query.
* Eq. 5  dynamic top-n budget, n = max(n_min, ceil(M * p)), with the
         n_local most recent blocks forced in by a +inf score.
* Algorithm 1  rectified sparse decoding: append, refresh block keys, and every
         f steps a dense re-encode of the last f tokens that overwrites their
         K/V and refreshes the block keys.
* Algorithm 2  split-K flash decoding over the selected blocks + combine
         (used here only as a self-check of the single-pass result).

Readings of the paper where it is silent or inconsistent (kept identical in
the CUDA path):

1. The ratio in Eq. 5 is the fraction of blocks KEPT (0.1 at "sparsity 0.9").
2. A masked key is removed from the softmax (score -inf), not multiplied by 0.
3. The pooled query is the mean of the g query heads of the group, taken
   before scoring; scores omit the 1/sqrt(d) factor (ranking-invariant).
4. The n_local forced blocks count inside n; n >= n_local and n <= M.
5. M = ceil(T / b) includes a partially filled last block, whose summary
   covers only its valid tokens. The current token is appended before
   selection, so it always attends to itself.
6. Ties in the top-n go to the lower block index.
7. ceil(M * p) is evaluated on the float64 product M * p.
8. After a rectification overwrite, touched blocks are recomputed from all of
   their tokens (a min/max cannot be "un-applied").
9. Rectified queries attend to the new (dense) K/V of the f tokens, causally:
   query i of the f sees positions [0, T - f + i].
10. Non-finite values (the paper assumes finite ones): a NaN among a block's
   valid keys makes that dimension of its Eq. 3 min and max NaN; a NaN
   summary element or pooled-query element makes the Eq. 4 score NaN; in
   Eq. 5 a NaN score ranks below every number, -inf included, and NaN scores
   tie among themselves (lower block index first). Forced local blocks score
   +inf whatever their summary holds.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

NEG_INF = -math.inf


def widen_bf16(bits) -> np.ndarray:
    """Exact bf16 (uint16 bit pattern) -> float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------
# Eq. 3 -- block representation
# --------------------------------------------------------------------------
def block_summaries(keys: np.ndarray, b: int):
    """Element-wise min and max of each block of b consecutive keys (Eq. 3).

    keys: [T, d] float64. Returns (kmin, kmax), each [M, d] with M = ceil(T/b);
    block i covers positions [i*b, min((i+1)*b, T)).
    """
    T, d = keys.shape
    M = (T + b - 1) // b
    kmin = np.empty((M, d))
    kmax = np.empty((M, d))
    for i in range(M):
        blk = keys[i * b:min((i + 1) * b, T)]
        kmin[i] = blk.min(axis=0)
        kmax[i] = blk.max(axis=0)
    return kmin, kmax


def online_summary_update(kmin_i, kmax_i, k_new, block_was_empty: bool):
    """Incremental Eq. 3 when one key joins block i (Section 2.1, online update)."""
    if block_was_empty:
        return k_new.copy(), k_new.copy()
    return np.minimum(kmin_i, k_new), np.maximum(kmax_i, k_new)


# --------------------------------------------------------------------------
# Eq. 4 / Eq. 5 -- block selection
# --------------------------------------------------------------------------
def pooled_query(q_group: np.ndarray) -> np.ndarray:
    """Average pooling of the g query heads of one GQA group (Section 2.1, Fig. 3)."""
    return q_group.mean(axis=0)


def quest_scores(q: np.ndarray, kmin: np.ndarray, kmax: np.ndarray) -> np.ndarray:
    """score_i = sum_j max(q_j * kmax_ij, q_j * kmin_ij)  (Eq. 4)."""
    return np.maximum(q[None, :] * kmax, q[None, :] * kmin).sum(axis=1)


def selection_budget(M: int, keep: float, n_min: int, n_local: int) -> int:
    """n = max(n_min, ceil(M * p)) (Eq. 5), then n_local <= n <= M (readings 4, 7)."""
    n = max(n_min, math.ceil(float(M) * float(keep)))
    n = max(n, n_local)
    return min(n, M)


def select_blocks(scores: np.ndarray, n: int, n_local: int) -> np.ndarray:
    """Top-n blocks after forcing the last n_local to +inf (Eq. 5 text).

    Ranking: higher score first, a NaN score below every number (reading 10),
    ties to the lower block index. Returns the selected block ids in
    ascending order.
    """
    M = scores.shape[0]
    s = scores.astype(np.float64).copy()
    if n_local > 0:
        s[max(0, M - n_local):] = math.inf
    nan = np.isnan(s)
    # primary: NaN last, then -score, then the block index
    order = np.lexsort((np.arange(M), np.where(nan, 0.0, -s), nan))
    return np.sort(order[:n])


# --------------------------------------------------------------------------
# Eq. 1 / Eq. 2 -- attention over a set of key positions
# --------------------------------------------------------------------------
def attend_positions(q: np.ndarray, K: np.ndarray, V: np.ndarray, positions: np.ndarray, scale: float):
    """softmax(q K_P^T * scale) V_P over the key positions P (Eq. 1 restricted).

    q: [g, d]; K, V: [T, d]; positions: int array. Returns (out [g, d], lse [g]),
    lse the natural log of the softmax denominator of the scaled logits. An
    empty P gives out = 0 and lse = -inf.
    """
    g, d = q.shape
    if positions.size == 0:
        return np.zeros((g, d)), np.full(g, NEG_INF)
    logits = (q @ K[positions].T) * scale          # [g, P]
    m = logits.max(axis=1, keepdims=True)
    e = np.exp(logits - m)
    den = e.sum(axis=1, keepdims=True)
    out = (e @ V[positions]) / den
    lse = (m + np.log(den))[:, 0]
    return out, lse


def attend_prefix(q: np.ndarray, K: np.ndarray, V: np.ndarray, n: int, scale: float):
    """attend_positions over the contiguous positions [0, n) (views, no gather)."""
    if n <= 0:
        g, d = q.shape
        return np.zeros((g, d)), np.full(g, NEG_INF)
    logits = (q @ K[:n].T) * scale
    m = logits.max(axis=1, keepdims=True)
    e = np.exp(logits - m)
    den = e.sum(axis=1, keepdims=True)
    return (e @ V[:n]) / den, (m + np.log(den))[:, 0]


def block_positions(blocks: np.ndarray, b: int, T: int) -> np.ndarray:
    """Key positions covered by the given blocks, restricted to [0, T)."""
    if len(blocks) == 0:
        return np.zeros(0, dtype=np.int64)
    pos = (np.asarray(blocks, dtype=np.int64)[:, None] * b + np.arange(b)[None, :]).reshape(-1)
    return pos[pos < T]


def gbsa_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, T: int, blocks: np.ndarray, b: int,
                   scale: float):
    """GBSA for one GQA group (Eq. 2): all g heads attend to the same blocks."""
    return attend_positions(q, K, V, block_positions(blocks, b, T), scale)


def dense_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, T: int, scale: float):
    """Dense attention over positions [0, T) (Eq. 1)."""
    return attend_prefix(q, K, V, T, scale)


def split_combine_attention(q, K, V, T, blocks, b, scale, num_splits: int):
    """Algorithm 2: split the selected blocks evenly over num_splits, attend
    each split separately, then combine the partials by their log-sum-exp."""
    blocks = np.asarray(blocks)
    n = len(blocks)
    per = (n + num_splits - 1) // num_splits if n else 0
    outs, lses = [], []
    for s in range(num_splits):
        part = blocks[s * per:min(n, (s + 1) * per)] if per else blocks[:0]
        o, l = gbsa_attention(q, K, V, T, part, b, scale)
        outs.append(o)
        lses.append(l)
    lses = np.stack(lses)                        # [S, g]
    outs = np.stack(outs)                        # [S, g, d]
    big = lses.max(axis=0)                       # [g]
    w = np.where(np.isfinite(lses), np.exp(lses - big[None, :]), 0.0)
    tot = w.sum(axis=0)
    out = (w[:, :, None] * outs).sum(axis=0) / tot[:, None]
    return out, big + np.log(tot)


# --------------------------------------------------------------------------
# Algorithm 1 -- per-sequence state and the two phases
# --------------------------------------------------------------------------
@dataclass
class ResaParams:
    keep: float
    n_min_blocks: int
    n_local_blocks: int
    block_size: int = 16
    scale: float | None = None        # None: 1/sqrt(d)

    def sm_scale(self, d: int) -> float:
        return 1.0 / math.sqrt(d) if self.scale is None else self.scale


class SequenceState:
    """KV cache and block key cache of one sequence (Algorithm 1's K and B).

    K, V: [Hkv, capacity, d] float64; kmin/kmax: [Hkv, capacity/b, d]; T = tokens.
    """

    def __init__(self, num_kv_heads: int, capacity: int, d: int, b: int):
        self.Hkv, self.d, self.b = num_kv_heads, d, b
        self.K = np.zeros((num_kv_heads, capacity, d))
        self.V = np.zeros((num_kv_heads, capacity, d))
        nb = (capacity + b - 1) // b
        self.kmin = np.zeros((num_kv_heads, nb, d))
        self.kmax = np.zeros((num_kv_heads, nb, d))
        self.T = 0

    def prefill(self, K0: np.ndarray, V0: np.ndarray):
        """Prefill: write the prompt's K/V and build every block summary."""
        T0 = K0.shape[1]
        self.K[:, :T0] = K0
        self.V[:, :T0] = V0
        self.T = T0
        self.refresh_blocks(0, (T0 + self.b - 1) // self.b)

    def refresh_blocks(self, first: int, last_excl: int):
        """Recompute block summaries [first, last_excl) from the valid tokens (Eq. 3)."""
        for h in range(self.Hkv):
            mn, mx = block_summaries(self.K[h, :self.T], self.b)
            self.kmin[h, first:last_excl] = mn[first:last_excl]
            self.kmax[h, first:last_excl] = mx[first:last_excl]

    def append(self, k: np.ndarray, v: np.ndarray):
        """Update KV cache and block key cache with one token (Algorithm 1)."""
        t = self.T
        i = t // self.b
        for h in range(self.Hkv):
            self.K[h, t] = k[h]
            self.V[h, t] = v[h]
            self.kmin[h, i], self.kmax[h, i] = online_summary_update(
                self.kmin[h, i], self.kmax[h, i], k[h], block_was_empty=(t % self.b == 0))
        self.T = t + 1

    def overwrite_tail(self, k_new: np.ndarray, v_new: np.ndarray):
        """Rectification write-back: the last f tokens' K/V are replaced by the
        dense ones and the touched block keys recomputed (Algorithm 1, reading 8).
        k_new, v_new: [f, Hkv, d]."""
        f = k_new.shape[0]
        t0 = self.T - f
        for h in range(self.Hkv):
            self.K[h, t0:self.T] = k_new[:, h]
            self.V[h, t0:self.T] = v_new[:, h]
        self.refresh_blocks(t0 // self.b, (self.T - 1) // self.b + 1)

    @property
    def num_blocks(self) -> int:
        return (self.T + self.b - 1) // self.b


def select_for_group(state: SequenceState, h: int, q_group: np.ndarray, p: ResaParams):
    """Pooled query -> Quest scores -> top-n (Eq. 4, Eq. 5) for KV head h."""
    M = state.num_blocks
    qbar = pooled_query(q_group)
    scores = quest_scores(qbar, state.kmin[h, :M], state.kmax[h, :M])
    n = selection_budget(M, p.keep, p.n_min_blocks, p.n_local_blocks)
    return select_blocks(scores, n, p.n_local_blocks), scores, n


def sparse_decode_step(state: SequenceState, q: np.ndarray, k: np.ndarray, v: np.ndarray, p: ResaParams):
    """One SparseForward of Algorithm 1 for one sequence, attention part.

    Order (reading 5): append the token's K/V and refresh its block key, then
    select blocks per GQA group from the pooled query, then GBSA.
    q: [Hq, d]; k, v: [Hkv, d]. Returns (out [Hq, d], lse [Hq], selected list
    per KV head, scores list per KV head).
    """
    state.append(k, v)
    Hq, d = q.shape
    g = Hq // state.Hkv
    scale = p.sm_scale(d)
    out = np.zeros((Hq, d))
    lse = np.zeros(Hq)
    sel, scs = [], []
    for h in range(state.Hkv):
        qg = q[h * g:(h + 1) * g]
        blocks, scores, _ = select_for_group(state, h, qg, p)
        o, l = gbsa_attention(qg, state.K[h], state.V[h], state.T, blocks, state.b, scale)
        out[h * g:(h + 1) * g] = o
        lse[h * g:(h + 1) * g] = l
        sel.append(blocks)
        scs.append(scores)
    return out, lse, sel, scs


def rectify_attention(q_new: np.ndarray, K: np.ndarray, V: np.ndarray, k_new: np.ndarray, v_new: np.ndarray,
                      T: int, scale: float):
    """Dense causal attention of the last f tokens (Section 2.2, reading 9).

    q_new: [f, Hq, d]; K, V: [Hkv, >=T, d] cache (positions < T - f are used);
    k_new, v_new: [f, Hkv, d], the new K/V of positions [T - f, T).
    Query row i (position T - f + i) attends to positions [0, T - f + i].
    Returns (out [f, Hq, d], lse [f, Hq]).
    """
    f, Hq, d = q_new.shape
    Hkv = K.shape[0]
    g = Hq // Hkv
    t0 = T - f
    out = np.zeros((f, Hq, d))
    lse = np.zeros((f, Hq))
    for h in range(Hkv):
        Kh = np.concatenate([K[h, :t0], k_new[:, h]], axis=0)   # [T, d]
        Vh = np.concatenate([V[h, :t0], v_new[:, h]], axis=0)
        for i in range(f):
            o, l = attend_prefix(q_new[i, h * g:(h + 1) * g], Kh, Vh, t0 + i + 1, scale)
            out[i, h * g:(h + 1) * g] = o
            lse[i, h * g:(h + 1) * g] = l
    return out, lse


def rectify_step(state: SequenceState, q_new, k_new, v_new, p: ResaParams):
    """DenseForward of the last f tokens, then overwrite their K/V and refresh
    the block keys (Algorithm 1, rectification branch)."""
    scale = p.sm_scale(q_new.shape[-1])
    out, lse = rectify_attention(q_new, state.K, state.V, k_new, v_new, state.T, scale)
    state.overwrite_tail(k_new, v_new)
    return out, lse


def memory_access_ratio(b: int, keep: float, f: int) -> float:
    """Average memory access per decode step relative to dense decoding (Eq. 6)."""
    return 1.0 / b + keep + 1.0 / f
