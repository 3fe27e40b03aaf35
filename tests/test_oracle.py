"""Pins of the fp64 oracle against things other than itself (CPU only).

Each test checks an oracle function against a hand-worked example
(tests/golden), a closed form, brute force on tiny inputs, or a library
routine (torch's fp64 scaled_dot_product_attention). They are chosen so that
a dropped term, a flipped sign, a wrong index or a transposed operand in the
oracle fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_04108_gb300 import synth

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "worked_examples.json")))


def rand_bf16(g, shape, scale=1.0):
    return O.widen_bf16(synth.normal_bf16(g, shape, scale))


def sdpa(q, K, V, scale, mask=None):
    """torch fp64 SDPA as the textbook reference. q [g,d], K/V [T,d]."""
    qt = torch.from_numpy(q)[:, None, :]                      # heads as batch, 1 query each
    Kt = torch.from_numpy(K)[None].expand(q.shape[0], -1, -1)
    Vt = torch.from_numpy(V)[None].expand(q.shape[0], -1, -1)
    am = None if mask is None else torch.from_numpy(mask)[:, None, :]
    out = torch.nn.functional.scaled_dot_product_attention(qt, Kt, Vt, attn_mask=am, scale=scale)
    return out[:, 0, :].numpy()


# ----------------------------------------------------------------- Eq. 3 ---
def test_summaries_worked_example():
    ex = GOLDEN["quest_block_score"]
    kmin, kmax = O.block_summaries(np.array(ex["keys"]), ex["block_size"])
    assert np.array_equal(kmin, np.array(ex["kmin"]))
    assert np.array_equal(kmax, np.array(ex["kmax"]))


@pytest.mark.parametrize("T,b", [(1, 16), (16, 16), (37, 16), (50, 7), (9, 1)])
def test_summaries_brute_force(T, b):
    g = synth.rng(11 + T)
    K = rand_bf16(g, (T, 5))
    kmin, kmax = O.block_summaries(K, b)
    M = (T + b - 1) // b
    assert kmin.shape == (M, 5)
    for i in range(M):
        for j in range(5):
            vals = [K[t, j] for t in range(T) if t // b == i]
            lo, hi = vals[0], vals[0]
            for v in vals[1:]:
                lo = v if v < lo else lo
                hi = v if v > hi else hi
            assert kmin[i, j] == lo and kmax[i, j] == hi


def test_online_update_equals_recompute():
    g = synth.rng(5)
    b, d, T = 16, 8, 70
    K = rand_bf16(g, (1, T, d))
    st = O.SequenceState(1, 80, d, b)
    st.prefill(K[:, :3], K[:, :3])
    for t in range(3, T):
        st.append(K[:, t], K[:, t])
    mn, mx = O.block_summaries(K[0], b)
    M = (T + b - 1) // b
    assert np.array_equal(st.kmin[0, :M], mn) and np.array_equal(st.kmax[0, :M], mx)


# ----------------------------------------------------------------- Eq. 4 ---
def test_pooling_and_score_worked_example():
    ex = GOLDEN["quest_block_score"]
    q = O.pooled_query(np.array(ex["q_heads"]))
    assert np.array_equal(q, np.array(ex["pooled_query"]))
    kmin, kmax = O.block_summaries(np.array(ex["keys"]), ex["block_size"])
    assert np.array_equal(O.quest_scores(q, kmin, kmax), np.array(ex["scores"]))


def test_score_is_upper_bound_of_every_key():
    g = synth.rng(21)
    for trial in range(20):
        b, d, T = 16, 32, 16 * 5 + (trial % 9)
        K = rand_bf16(g, (T, d), scale=1.0 + trial)
        q = g.standard_normal(d)
        kmin, kmax = O.block_summaries(K, b)
        s = O.quest_scores(q, kmin, kmax)
        for t in range(T):
            assert K[t] @ q <= s[t // b] + 1e-9 * (1 + abs(s[t // b]))
        # the bound is attained by the block's "corner" key
        for i in range(len(s)):
            corner = np.where(q >= 0, kmax[i], kmin[i])
            assert math.isclose(corner @ q, s[i], rel_tol=1e-12, abs_tol=1e-12)


def test_score_single_token_blocks_equal_dot_product():
    g = synth.rng(3)
    K = rand_bf16(g, (9, 16))
    q = g.standard_normal(16)
    kmin, kmax = O.block_summaries(K, 1)
    assert np.allclose(O.quest_scores(q, kmin, kmax), K @ q, rtol=0, atol=1e-12)


# ----------------------------------------------------------------- Eq. 5 ---
@pytest.mark.parametrize("case", GOLDEN["budget"]["cases"], ids=lambda c: f"M{c['M']}")
def test_budget_worked(case):
    assert O.selection_budget(case["M"], case["keep"], case["n_min"], case["n_local"]) == case["n"]


def test_topn_worked_example():
    ex = GOLDEN["top_n_with_local"]
    got = O.select_blocks(np.array(ex["scores"]), ex["n"], ex["n_local"])
    assert got.tolist() == ex["selected"]


def test_topn_brute_force_count_of_better_blocks():
    """A block is kept iff fewer than n blocks beat it (higher forced score, or
    equal score and lower index): an independent statement of the rule."""
    g = synth.rng(8)
    for trial in range(200):
        M = int(g.integers(1, 14))
        scores = np.round(g.standard_normal(M) * 2) / 2          # many ties
        n_local = int(g.integers(0, 4))
        n = int(g.integers(max(1, min(n_local, M)), M + 1))
        forced = [i >= M - n_local for i in range(M)]
        eff = [math.inf if forced[i] else scores[i] for i in range(M)]
        want = []
        for i in range(M):
            better = sum(1 for j in range(M) if eff[j] > eff[i] or (eff[j] == eff[i] and j < i))
            if better < n:
                want.append(i)
        assert O.select_blocks(scores, n, n_local).tolist() == want


def test_topn_exhaustive_subset_maximises_score_sum():
    g = synth.rng(9)
    for trial in range(40):
        M, n = 8, 3
        scores = g.standard_normal(M)
        best = max(itertools.combinations(range(M), n), key=lambda c: sum(scores[list(c)]))
        assert O.select_blocks(scores, n, 0).tolist() == sorted(best)


# ------------------------------------------- non-finite values (reading 10) ---
def test_summary_nan_key_poisons_only_its_dimension():
    """A NaN key makes its block's min and max NaN in that dimension only; the
    online update agrees with the recompute (brute force over the other dims)."""
    g = synth.rng(71)
    b, d, T = 16, 6, 40
    K = rand_bf16(g, (T, d))
    K[20, 2] = np.nan                     # block 1, dimension 2
    kmin, kmax = O.block_summaries(K, b)
    for i in range(3):
        for j in range(d):
            vals = K[i * b:min(T, (i + 1) * b), j]
            if i == 1 and j == 2:
                assert np.isnan(kmin[i, j]) and np.isnan(kmax[i, j])
            else:
                assert kmin[i, j] == min(vals.tolist()) and kmax[i, j] == max(vals.tolist())
    st = O.SequenceState(1, 48, d, b)
    for t in range(T):
        st.append(K[None, t], K[None, t])
    assert np.array_equal(st.kmin[0, :3], kmin, equal_nan=True)
    assert np.array_equal(st.kmax[0, :3], kmax, equal_nan=True)


def test_score_nan_from_summary_or_query():
    g = synth.rng(72)
    kmin, kmax = O.block_summaries(rand_bf16(g, (64, 8)), 16)
    q = g.standard_normal(8)
    kmin[2, 5] = np.nan
    s = O.quest_scores(q, kmin, kmax)
    assert np.isnan(s[2]) and np.isfinite(np.delete(s, 2)).all()
    q[0] = np.nan
    assert np.isnan(O.quest_scores(q, kmin, kmax)).all()


def test_topn_nan_ranks_last_brute_force():
    """A block is kept iff fewer than n blocks beat it, where a number beats
    NaN, a larger number beats a smaller one, and within equal scores (NaN
    with NaN included) the lower index wins; forced blocks score +inf."""
    g = synth.rng(73)
    for trial in range(300):
        M = int(g.integers(1, 14))
        scores = np.round(g.standard_normal(M) * 2) / 2
        scores[g.random(M) < 0.3] = np.nan
        scores[g.random(M) < 0.1] = -np.inf
        n_local = int(g.integers(0, 4))
        n = int(g.integers(max(1, min(n_local, M)), M + 1))
        eff = [math.inf if i >= M - n_local else scores[i] for i in range(M)]

        def beats(j, i):
            a, c = eff[j], eff[i]
            if math.isnan(a) or math.isnan(c):
                return (not math.isnan(a)) or (math.isnan(c) and j < i)
            return a > c or (a == c and j < i)
        want = [i for i in range(M) if sum(1 for j in range(M) if j != i and beats(j, i)) < n]
        assert O.select_blocks(scores, n, n_local).tolist() == want


# --------------------------------------------------------- Eq. 1 / Eq. 2 ---
def test_two_key_softmax_worked():
    ex = GOLDEN["two_key_softmax"]
    out, lse = O.dense_attention(np.array(ex["q"]), np.array(ex["keys"]), np.array(ex["values"]), 2,
                                 1 / math.sqrt(2))
    assert np.allclose(out, np.array(ex["out"]), rtol=0, atol=1e-14)
    assert np.allclose(lse, np.array(ex["lse"]), rtol=0, atol=1e-14)


@pytest.mark.parametrize("T", [1, 17, 64, 200])
def test_dense_attention_matches_torch_sdpa(T):
    g = synth.rng(100 + T)
    q, K, V = rand_bf16(g, (7, 128)), rand_bf16(g, (T, 128)), rand_bf16(g, (T, 128))
    sc = 1 / math.sqrt(128)
    out, lse = O.dense_attention(q, K, V, T, sc)
    assert np.allclose(out, sdpa(q, K, V, sc), rtol=0, atol=1e-12)
    ref_lse = torch.logsumexp(torch.from_numpy(q @ K.T * sc), dim=1).numpy()
    assert np.allclose(lse, ref_lse, rtol=0, atol=1e-12)


def test_gbsa_all_blocks_equals_dense():
    """Check 1: sparse attention with every block selected is dense attention."""
    g = synth.rng(7)
    T, b = 77, 16
    q, K, V = rand_bf16(g, (4, 128)), rand_bf16(g, (T, 128)), rand_bf16(g, (T, 128))
    sc = 1 / math.sqrt(128)
    o, _ = O.gbsa_attention(q, K, V, T, np.arange((T + b - 1) // b), b, sc)
    assert np.allclose(o, sdpa(q, K, V, sc), rtol=0, atol=1e-12)


def test_gbsa_masks_unselected_and_out_of_range_keys():
    g = synth.rng(70)
    T, b = 70, 16                     # 5 blocks, last one holds 6 valid tokens
    q, K, V = rand_bf16(g, (3, 64)), rand_bf16(g, (80, 64)), rand_bf16(g, (80, 64))
    sc = 0.125
    blocks = np.array([1, 4])
    mask = np.zeros((3, 80), dtype=bool)
    for p in range(80):
        mask[:, p] = (p // b in (1, 4)) and p < T
    o, _ = O.gbsa_attention(q, K, V, T, blocks, b, sc)
    assert np.allclose(o, sdpa(q, K, V, sc, mask), rtol=0, atol=1e-12)


def test_gbsa_constant_keys_give_mean_value():
    g = synth.rng(71)
    T, b = 64, 16
    K = np.tile(rand_bf16(g, (1, 32)), (T, 1))
    V = rand_bf16(g, (T, 32))
    q = rand_bf16(g, (2, 32))
    blocks = np.array([0, 2])
    o, lse = O.gbsa_attention(q, K, V, T, blocks, b, 0.3)
    pos = np.r_[0:16, 32:48]
    assert np.allclose(o, V[pos].mean(axis=0)[None], rtol=0, atol=1e-12)
    assert np.allclose(lse, (q @ K[0]) * 0.3 + math.log(32), rtol=0, atol=1e-12)


def test_single_block_textbook_loop():
    g = synth.rng(72)
    b, d = 16, 8
    K, V, q = rand_bf16(g, (48, d)), rand_bf16(g, (48, d)), rand_bf16(g, (1, d))
    o, _ = O.gbsa_attention(q, K, V, 48, np.array([2]), b, 0.5)
    logits = [sum(q[0, j] * K[32 + t, j] for j in range(d)) * 0.5 for t in range(16)]
    mx = max(logits)
    w = [math.exp(x - mx) for x in logits]
    tot = sum(w)
    want = [sum(w[t] * V[32 + t, j] for t in range(16)) / tot for j in range(d)]
    assert np.allclose(o[0], want, rtol=0, atol=1e-12)


@pytest.mark.parametrize("splits", [1, 2, 3, 7, 20, 64])
def test_split_combine_equals_single_pass(splits):
    """Check 4 (Algorithm 2): softmax split-merge equals single-pass softmax,
    including splits that receive no block."""
    g = synth.rng(splits)
    T, b = 300, 16
    q, K, V = rand_bf16(g, (7, 128)), rand_bf16(g, (T, 128)), rand_bf16(g, (T, 128))
    blocks = np.sort(g.choice((T + b - 1) // b, 11, replace=False))
    o1, l1 = O.gbsa_attention(q, K, V, T, blocks, b, 0.088)
    o2, l2 = O.split_combine_attention(q, K, V, T, blocks, b, 0.088, splits)
    assert np.allclose(o1, o2, rtol=0, atol=1e-12) and np.allclose(l1, l2, rtol=0, atol=1e-12)


# -------------------------------------------------------- Algorithm 1 -------
def test_rectify_rows_match_causal_sdpa():
    g = synth.rng(80)
    Hkv, gq, d, T, f = 2, 3, 64, 53, 8
    K, V = rand_bf16(g, (Hkv, 60, d)), rand_bf16(g, (Hkv, 60, d))
    kn, vn = rand_bf16(g, (f, Hkv, d)), rand_bf16(g, (f, Hkv, d))
    qn = rand_bf16(g, (f, Hkv * gq, d))
    sc = 1 / 8
    out, _ = O.rectify_attention(qn, K, V, kn, vn, T, sc)
    for h in range(Hkv):
        Kf = np.concatenate([K[h, :T - f], kn[:, h]])
        Vf = np.concatenate([V[h, :T - f], vn[:, h]])
        # causal mask of the f new rows against T keys
        mask = np.arange(T)[None, :] <= (T - f + np.arange(f))[:, None]     # [f, T]
        for j in range(gq):
            qh = qn[:, h * gq + j]                                           # [f, d]
            qt = torch.from_numpy(qh)[None]
            ref = torch.nn.functional.scaled_dot_product_attention(
                qt, torch.from_numpy(Kf)[None], torch.from_numpy(Vf)[None],
                attn_mask=torch.from_numpy(mask)[None], scale=sc)[0].numpy()
            assert np.allclose(out[:, h * gq + j], ref, rtol=0, atol=1e-12)


def test_rectify_last_row_is_dense_decode():
    g = synth.rng(81)
    d, T, f = 32, 40, 4
    K, V = rand_bf16(g, (1, T, d)), rand_bf16(g, (1, T, d))
    kn, vn, qn = rand_bf16(g, (f, 1, d)), rand_bf16(g, (f, 1, d)), rand_bf16(g, (f, 2, d))
    out, _ = O.rectify_attention(qn, K, V, kn, vn, T, 0.2)
    Kf = np.concatenate([K[0, :T - f], kn[:, 0]])
    Vf = np.concatenate([V[0, :T - f], vn[:, 0]])
    assert np.allclose(out[-1], sdpa(qn[-1], Kf, Vf, 0.2), rtol=0, atol=1e-12)


@pytest.mark.parametrize("T0,f", [(64, 8), (37, 8), (100, 32), (5, 16)])
def test_rectified_cache_equals_dense_cache(T0, f):
    """Check 2: after the rectification write-back, KV cache and block keys
    equal those of decoding with the dense K/V from the start."""
    g = synth.rng(T0 * 100 + f)
    Hkv, d, b = 2, 16, 16
    cap = T0 + f + 16
    K0, V0 = rand_bf16(g, (Hkv, T0, d)), rand_bf16(g, (Hkv, T0, d))
    dk, dv = rand_bf16(g, (f, Hkv, d)), rand_bf16(g, (f, Hkv, d))
    sk, sv = dk + 0.05 * g.standard_normal(dk.shape), dv + 0.05 * g.standard_normal(dv.shape)
    a, c = O.SequenceState(Hkv, cap, d, b), O.SequenceState(Hkv, cap, d, b)
    a.prefill(K0, V0)
    c.prefill(K0, V0)
    for i in range(f):
        a.append(sk[i], sv[i])
        c.append(dk[i], dv[i])
    a.overwrite_tail(dk, dv)
    assert a.T == c.T
    assert np.array_equal(a.K, c.K) and np.array_equal(a.V, c.V)
    M = c.num_blocks
    assert np.array_equal(a.kmin[:, :M], c.kmin[:, :M]) and np.array_equal(a.kmax[:, :M], c.kmax[:, :M])
    # and both equal a from-scratch Eq. 3 over the dense keys
    for h in range(Hkv):
        mn, mx = O.block_summaries(c.K[h, :c.T], b)
        assert np.array_equal(a.kmin[h, :M], mn) and np.array_equal(a.kmax[h, :M], mx)


def test_decode_step_order_and_self_attention():
    """The appended token is selectable (forced local block) and attended."""
    g = synth.rng(90)
    Hkv, gq, d, b = 1, 2, 16, 16
    st = O.SequenceState(Hkv, 200, d, b)
    st.prefill(rand_bf16(g, (Hkv, 100, d)), rand_bf16(g, (Hkv, 100, d)))
    p = O.ResaParams(keep=0.0, n_min_blocks=1, n_local_blocks=1)
    k, v = rand_bf16(g, (Hkv, d)), rand_bf16(g, (Hkv, d))
    q = rand_bf16(g, (gq, d))
    out, _, sel, _ = O.sparse_decode_step(st, q, k, v, p)
    assert st.T == 101 and sel[0].tolist() == [6]     # only the forced last block (positions 96..100)
    Kb = st.K[0, 96:101]
    Vb = st.V[0, 96:101]
    assert np.allclose(out, sdpa(q, Kb, Vb, 0.25), rtol=0, atol=1e-12)


def test_memory_access_ratio_worked():
    ex = GOLDEN["memory_access_ratio"]
    assert math.isclose(O.memory_access_ratio(ex["b"], ex["keep"], ex["f"]), ex["ratio"], rel_tol=1e-15)


def test_widen_bf16_exact():
    bits = np.array([0x3F80, 0xBF80, 0x4049, 0x0000, 0x8000, 0x7F7F], dtype=np.uint16)
    want = [1.0, -1.0, 3.140625, 0.0, -0.0, 3.3895313892515355e38]
    assert O.widen_bf16(bits).tolist() == want
