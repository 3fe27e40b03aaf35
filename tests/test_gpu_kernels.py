"""Per-call parity of the CUDA path (through the C ABI) against the fp64 oracle
on seeded inputs: cache commit / summaries (bit-exact), block selection
(exact up to the near-tie rule), sparse decode and rectification (2e-2
max-abs, 1e-3 mean-abs), plus device-side error reporting."""
import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_04108_gb300 import resa, synth
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu


def seq_inputs(seed, B, Hkv, lens, d=128, k_scale=1.0):
    g = synth.rng(seed)
    Ks = [synth.normal_bf16(g, (Hkv, T, d), k_scale) for T in lens]
    Vs = [synth.normal_bf16(g, (Hkv, T, d)) for T in lens]
    return Ks, Vs


# ---------------------------------------------------------------- Eq. 3 ---
@pytest.mark.parametrize("lens", [[16], [1, 17, 100, 333], [4096, 4095]])
def test_update_summaries_bit_exact(lens):
    Hkv = 2
    Ks, Vs = seq_inputs(1, len(lens), Hkv, lens)
    maxb = (max(lens) + 15) // 16 + 3
    cache = H.make_cache(Ks, Vs, Hkv * 4, maxb, zero_pools=False)
    summ = H.host_f64(cache.summaries)          # [B, Hkv, maxb, 2, d]
    for b, T in enumerate(lens):
        M = (T + 15) // 16
        for h in range(Hkv):
            mn, mx = O.block_summaries(O.widen_bf16(Ks[b][h]), 16)
            assert np.array_equal(summ[b, h, :M, 0], mn)
            assert np.array_equal(summ[b, h, :M, 1], mx)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)


def test_update_summaries_range_only_touches_range():
    Ks, Vs = seq_inputs(2, 1, 1, [200])
    cache = H.make_cache(Ks, Vs, 2, 16)
    cache.summaries.zero_()
    resa.resa_update_summaries(cache.struct, 3, 7)
    s = H.host_f64(cache.summaries)[0, 0]
    mn, mx = O.block_summaries(O.widen_bf16(Ks[0][0]), 16)
    assert np.all(s[:3] == 0) and np.all(s[7:] == 0)
    assert np.array_equal(s[3:7, 0], mn[3:7]) and np.array_equal(s[3:7, 1], mx[3:7])


@pytest.mark.parametrize("lens,n_new", [([30, 16, 1], 1), ([30, 47, 64], 5), ([0, 15, 16], 20)])
def test_commit_append_matches_oracle(lens, n_new):
    Hkv, d = 2, 128
    Ks, Vs = seq_inputs(3, len(lens), Hkv, lens)
    maxb = 8
    cache = H.make_cache(Ks, Vs, 4, maxb)
    g = synth.rng(33)
    kn = synth.normal_bf16(g, (len(lens), n_new, Hkv, d))
    vn = synth.normal_bf16(g, (len(lens), n_new, Hkv, d))
    resa.resa_commit_kv(cache.struct, H.dev_bf16(kn), H.dev_bf16(vn), n_new, False)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    summ = H.host_f64(cache.summaries)
    for b, T in enumerate(lens):
        st = H.oracle_state(Ks[b], Vs[b], maxb * 16)
        for t in range(n_new):
            st.append(O.widen_bf16(kn[b, t]), O.widen_bf16(vn[b, t]))
        assert int(cache.seq_lens[b]) == T + n_new
        K, V = H.logical_kv(cache, b)
        assert np.array_equal(O.widen_bf16(K), st.K[:, :st.T]) and np.array_equal(O.widen_bf16(V), st.V[:, :st.T])
        M = st.num_blocks
        assert np.array_equal(summ[b, :, :M, 0], st.kmin[:, :M]) and np.array_equal(summ[b, :, :M, 1], st.kmax[:, :M])


@pytest.mark.parametrize("lens,f", [([64, 100], 8), ([37, 333], 32), ([64, 200], 64), ([16, 17], 16)])
def test_commit_overwrite_matches_oracle(lens, f):
    Hkv, d = 4, 128
    Ks, Vs = seq_inputs(4, len(lens), Hkv, lens)
    maxb = 24
    cache = H.make_cache(Ks, Vs, 28, maxb)
    g = synth.rng(44)
    kn = synth.normal_bf16(g, (len(lens), f, Hkv, d))
    vn = synth.normal_bf16(g, (len(lens), f, Hkv, d))
    resa.resa_commit_kv(cache.struct, H.dev_bf16(kn), H.dev_bf16(vn), f, True)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    summ = H.host_f64(cache.summaries)
    for b, T in enumerate(lens):
        st = H.oracle_state(Ks[b], Vs[b], maxb * 16)
        st.overwrite_tail(O.widen_bf16(kn[b]), O.widen_bf16(vn[b]))
        assert int(cache.seq_lens[b]) == T
        K, V = H.logical_kv(cache, b)
        assert np.array_equal(O.widen_bf16(K), st.K[:, :T]) and np.array_equal(O.widen_bf16(V), st.V[:, :T])
        M = st.num_blocks
        assert np.array_equal(summ[b, :, :M, 0], st.kmin[:, :M]) and np.array_equal(summ[b, :, :M, 1], st.kmax[:, :M])


# ---------------------------------------------------------- Eq. 4 / 5 -----
def run_select(cache, q_bits, p, n_cap):
    B, Hkv = cache.batch, cache.Hkv
    idx = torch.empty((B, Hkv, n_cap), dtype=torch.int32, device="cuda")
    cnt = torch.empty((B, Hkv), dtype=torch.int32, device="cuda")
    ws, nb = H.workspace(cache, n_cap)
    resa.resa_select_blocks(cache.struct, H.dev_bf16(q_bits), p, idx, cnt, n_cap, ws, nb)
    return idx.cpu().numpy(), cnt.cpu().numpy()


# Caches of up to 6144 blocks per sequence take the one-CTA top-n, larger ones
# the cluster top-n: `wide` pads the page-table row past that bound so that
# every case runs through both.
@pytest.mark.parametrize("wide", [False, True])
@pytest.mark.parametrize("g,Hkv,lens,keep,n_min,n_local", [
    (4, 2, [4100], 0.1, 16, 4),            # the 4K workload shape
    (7, 4, [1000, 2053, 37, 16], 0.1, 8, 1),
    (1, 1, [513], 0.25, 0, 0),
    (8, 1, [300, 5000], 0.05, 3, 2),
    (7, 4, [100, 80], 0.5, 16, 1),         # M <= n: every block selected
    (2, 2, [160], 0.0, 0, 12),             # n_local >= n
    (3, 2, [300, 900], 0.2, 4, 1),         # group sizes 3, 5, 6: the pooled query's
    (5, 2, [700], 0.2, 4, 1),              # head sum is split over four lane groups
    (6, 1, [1200], 0.1, 0, 2),             # (heads j and j + 4)
])
def test_select_matches_oracle(g, Hkv, lens, keep, n_min, n_local, wide):
    Ks, Vs = seq_inputs(5 + len(lens), len(lens), Hkv, lens)
    maxb = max((T + 15) // 16 for T in lens) + 4
    if wide:
        maxb = max(maxb, 6200)
    cache = H.make_cache(Ks, Vs, g * Hkv, maxb, compact=wide)
    gq = synth.rng(55)
    q = synth.normal_bf16(gq, (len(lens), g * Hkv, 128))
    p = resa.params(keep, n_min, n_local)
    n_cap = resa.resa_max_selected(cache.struct, p) + 3
    idx, cnt = run_select(cache, q, p, n_cap)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    for b, T in enumerate(lens):
        st = H.oracle_state(Ks[b], Vs[b], maxb * 16)
        for h in range(Hkv):
            sel, scores, n = O.select_for_group(st, h, O.widen_bf16(q[b, h * g:(h + 1) * g]),
                                                O.ResaParams(keep, n_min, n_local))
            assert cnt[b, h] == n
            assert np.all(idx[b, h, n:] == -1)
            H.check_selection(idx[b, h, :n], scores, n, n_local)


def check_select_case(cache, Ks, Vs, q, p, maxb, idx, cnt):
    g = cache.Hq // cache.Hkv
    for b, Kb in enumerate(Ks):
        st = H.oracle_state(Kb, Vs[b], maxb * 16)
        for h in range(cache.Hkv):
            sel, scores, n = O.select_for_group(st, h, O.widen_bf16(q[b, h * g:(h + 1) * g]),
                                                O.ResaParams(p.keep_ratio, p.n_min_blocks, p.n_local_blocks))
            assert cnt[b, h] == n
            assert np.all(idx[b, h, n:] == -1)
            H.check_selection(idx[b, h, :n], scores, n, p.n_local_blocks)


@pytest.mark.parametrize("maxb", [72, 6150])  # one-CTA and cluster top-n
def test_select_many_small_units_and_repeat(maxb):
    """More (sequence, KV head) units than SMs, of one or two score pieces
    each, ragged lengths and two empty sequences (count 0, ids -1). A second
    call on the same state must give the same result."""
    B, Hkv, g = 100, 2, 4
    lens = [int(x) for x in synth.rng(71).integers(1, 1100, size=B)]
    lens[3] = 0
    lens[50] = 0
    Ks, Vs = seq_inputs(72, B, Hkv, lens)
    cache = H.make_cache(Ks, Vs, g * Hkv, maxb, compact=True)
    q = synth.normal_bf16(synth.rng(73), (B, g * Hkv, 128))
    p = resa.params(0.2, 2, 1)
    n_cap = resa.resa_max_selected(cache.struct, p)
    idx, cnt = run_select(cache, q, p, n_cap)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    check_select_case(cache, Ks, Vs, q, p, maxb, idx, cnt)
    idx2, cnt2 = run_select(cache, q, p, n_cap)
    assert np.array_equal(idx, idx2) and np.array_equal(cnt, cnt2)


def test_select_large_unit():
    """One unit of 30,001 blocks (3,751 keys staged per CTA of the cluster)."""
    M = 30001
    T = M * 16 - 7
    Ks, Vs = seq_inputs(74, 1, 1, [T])
    maxb = M + 3
    cache = H.make_cache(Ks, Vs, 2, maxb)
    q = synth.normal_bf16(synth.rng(75), (1, 2, 128))
    p = resa.params(0.05, 16, 4)
    n_cap = resa.resa_max_selected(cache.struct, p)
    idx, cnt = run_select(cache, q, p, n_cap)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    check_select_case(cache, Ks, Vs, q, p, maxb, idx, cnt)


def test_select_at_the_largest_cache():
    """One unit of 409,600 blocks (6.55M tokens), the largest page-table row
    the library accepts: the cluster top-n stages 51,200 keys per CTA (its
    whole 200 KB). Every block holds one key repeated, so its summary is
    that key on both sides (checked bit for bit); the ids equal the oracle's
    up to the near-tie rule."""
    M, g, Hkv = 409600, 2, 1
    T = M * 16 - 5
    keys = synth.normal_bf16(synth.rng(81), (M, 128))
    pt = synth.page_table(synth.rng(82), 1, M)
    cache = resa.PagedKVCache(1, g * Hkv, Hkv, M, pt, zero_pools=True)
    rows = torch.from_numpy(pt[0].astype(np.int64)).cuda()
    cache.k_pool.view(M, 16, 128)[rows] = H.dev_bf16(keys)[:, None, :].expand(M, 16, 128)
    cache.seq_lens.fill_(T)
    resa.resa_update_summaries(cache.struct, 0, -1)
    summ = H.host_bits(cache.summaries)[0, 0]
    assert np.array_equal(summ[:, 0], keys) and np.array_equal(summ[:, 1], keys)
    q = synth.normal_bf16(synth.rng(83), (1, g, 128))
    p = resa.params(0.05, 128, 1)
    n_cap = resa.resa_max_selected(cache.struct, p)
    idx, cnt = run_select(cache, q, p, n_cap)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    kf = O.widen_bf16(keys)
    scores = O.quest_scores(O.pooled_query(O.widen_bf16(q[0])), kf, kf)
    n = O.selection_budget(M, 0.05, 128, 1)
    assert cnt[0, 0] == n == 20480
    assert np.all(idx[0, 0, n:] == -1)
    H.check_selection(idx[0, 0, :n], scores, n, 1)


@pytest.mark.parametrize("M", [6144, 5121, 4000])
def test_select_one_cta_at_its_size_bound(M):
    """The one-CTA top-n at the largest cache it serves: 6144 blocks fill all
    twelve key slots of every thread; 5121 blocks leave the last warp with no
    ids and the one before it with a partial range; 4000 blocks take the
    8-slot instantiation. Some blocks repeat, so
    ties at the boundary are resolved by index."""
    T = M * 16 - 5
    gk = synth.rng(76)
    K = synth.normal_bf16(gk, (1, T, 128))
    K[:, 16 * 100:16 * 400] = np.tile(K[:, 16 * 99:16 * 100], (1, 300, 1))   # 300 identical blocks
    V = synth.normal_bf16(gk, (1, T, 128))
    cache = H.make_cache([K], [V], 7, M)
    q = synth.normal_bf16(synth.rng(77), (1, 7, 128))
    p = resa.params(0.1, 16, 2)
    n_cap = resa.resa_max_selected(cache.struct, p)
    idx, cnt = run_select(cache, q, p, n_cap)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    check_select_case(cache, [K], [V], q, p, M, idx, cnt)


@pytest.mark.parametrize("maxb", [44, 6200])  # one-CTA and cluster top-n
def test_select_ties_go_to_lower_index(maxb):
    """Identical blocks give identical scores; the lower ids must win."""
    Hkv, g, T = 1, 4, 16 * 40
    blk = synth.normal_bf16(synth.rng(6), (Hkv, 16, 128))
    K = np.tile(blk, (1, 40, 1))
    V = synth.normal_bf16(synth.rng(7), (Hkv, T, 128))
    cache = H.make_cache([K], [V], g, maxb, compact=True)
    q = synth.normal_bf16(synth.rng(8), (1, g, 128))
    p = resa.params(0.1, 0, 1)
    idx, cnt = run_select(cache, q, p, 16)
    assert cnt[0, 0] == 4
    assert idx[0, 0, :4].tolist() == [0, 1, 2, 39]


def _tied_unit(M, tied, scale, seed):
    """Keys of one KV head: M random blocks, with the blocks `tied` replaced
    by one shared block scaled by `scale` (identical summaries, so identical
    scores in the oracle and on the GPU)."""
    K = synth.normal_bf16(synth.rng(seed), (1, M * 16, 128))
    blk = synth.normal_bf16(synth.rng(seed + 1), (1, 16, 128), scale)
    for m in tied:
        K[:, m * 16:(m + 1) * 16] = blk
    V = synth.normal_bf16(synth.rng(seed + 2), (1, M * 16, 128))
    return K, V


@pytest.mark.parametrize("tied,scale,keep", [
    (range(700, 1300), 4.0, 0.04),   # 600 top-scoring equal blocks over two CTAs: the boundary bucket is gathered
    (range(0, 6397), 1.0, 0.1),      # ~6,400 equal blocks at the boundary: exchanged passes and counts
])
def test_select_cluster_ties_at_the_boundary(tied, scale, keep):
    """Cluster top-n (6,400 blocks, 800 per CTA) with the n-th largest score
    shared by many blocks: the ids equal the oracle's exactly, ties to the
    lower ids across CTAs."""
    M, g = 6400, 4
    K, V = _tied_unit(M, tied, scale, 91)
    maxb = M + 10
    cache = H.make_cache([K], [V], g, maxb, compact=True)
    q = synth.normal_bf16(synth.rng(95), (1, g, 128))
    p = resa.params(keep, 0, 1)
    n_cap = resa.resa_max_selected(cache.struct, p)
    idx, cnt = run_select(cache, q, p, n_cap)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    st = H.oracle_state(K, V, maxb * 16)
    _, scores, n = O.select_for_group(st, 0, O.widen_bf16(q[0]), O.ResaParams(keep, 0, 1))
    assert cnt[0, 0] == n
    tie = scores[tied[0]]
    assert np.sum(scores > tie) < n - 1 < np.sum(scores >= tie)  # the boundary lies inside the tied blocks
    assert np.array_equal(idx[0, 0, :n], O.select_blocks(scores, n, 1))


@pytest.mark.parametrize("n_tied,n", [(20, 11), (32, 17), (100, 51)])
def test_select_one_cta_ties_at_the_boundary(n_tied, n):
    """One-CTA top-n (2,048 blocks, the 32K shape) with the n-th largest
    score shared by a group of 20, 32 or 100 equal top-scoring blocks (alone
    in the first radix pass's top bucket): the ids equal the oracle's
    exactly, ties to the lower ids."""
    M, g = 2048, 4
    tied = range(300, 300 + 3 * n_tied, 3)
    K, V = _tied_unit(M, tied, 4.0, 71)
    maxb = M + 10
    cache = H.make_cache([K], [V], g, maxb, compact=True)
    q = synth.normal_bf16(synth.rng(75), (1, g, 128))
    keep = n / M  # exact in binary: ceil(M keep) = n
    p = resa.params(keep, 0, 1)
    n_cap = resa.resa_max_selected(cache.struct, p)
    idx, cnt = run_select(cache, q, p, n_cap)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    st = H.oracle_state(K, V, maxb * 16)
    _, scores, n_o = O.select_for_group(st, 0, O.widen_bf16(q[0]), O.ResaParams(keep, 0, 1))
    assert cnt[0, 0] == n_o == n
    tie = scores[tied[0]]
    assert np.sum(scores > tie) < n - 1 < np.sum(scores >= tie)  # the boundary lies inside the tied blocks
    assert np.array_equal(idx[0, 0, :n], O.select_blocks(scores, n, 1))


@pytest.mark.parametrize("maxb", [110, 6200])  # one-CTA and cluster top-n
def test_select_budget_over_cap_is_reported_and_clamped(maxb):
    Ks, Vs = seq_inputs(9, 1, 1, [1600])
    cache = H.make_cache(Ks, Vs, 2, maxb, compact=True)
    q = synth.normal_bf16(synth.rng(9), (1, 2, 128))
    p = resa.params(0.1, 0, 1)
    idx, cnt = run_select(cache, q, p, 5)               # n = 10 > n_cap = 5
    code, _ = resa.resa_read_device_error(cache.struct)
    assert code == 3 and cnt[0, 0] == 5
    assert len(set(idx[0, 0].tolist())) == 5


# ------------------------------------------ fused decode step (Alg. 1) ----
def _decode_step_caches(lens, Hkv, g, maxb, reserve, seed):
    Ks, Vs = seq_inputs(seed, len(lens), Hkv, lens)
    mk = lambda: H.make_cache(Ks, Vs, g * Hkv, maxb, zero_pools=True, compact=True, reserve_blocks=reserve)
    return mk(), mk()


@pytest.mark.parametrize("wide", [False, True])  # one-CTA / cluster top-n
def test_decode_step_equals_commit_select_decode(wide):
    """resa_decode_step gives, bit for bit, what resa_commit_kv(append 1) +
    resa_select_blocks + resa_sparse_decode give: ids, counts, outputs and
    log-sum-exps every step, and the same pools, summaries and lengths after.
    The ragged lengths put the appended token at every offset of its block
    over 20 steps (T % 16 = 15 fills a block, 0 opens one); one sequence
    starts empty."""
    B, Hkv, g, steps = 4, 2, 4, 20
    lens = [31, 0, 500, 1000]
    maxb = 6200 if wide else (max(lens) + steps + 15) // 16 + 2
    A, F = _decode_step_caches(lens, Hkv, g, maxb, (steps + 15) // 16 + 1, 91)
    p = resa.params(0.2, 2, 1)
    n_cap = resa.resa_max_selected(A.struct, p)
    wa, nb = H.workspace(A, n_cap)
    wf, _ = H.workspace(F, n_cap)
    mk = lambda shape, dt: torch.empty(shape, dtype=dt, device="cuda")
    ia, ifu = mk((B, Hkv, n_cap), torch.int32), mk((B, Hkv, n_cap), torch.int32)
    ca, cf = mk((B, Hkv), torch.int32), mk((B, Hkv), torch.int32)
    oa, of = mk((B, g * Hkv, 128), torch.bfloat16), mk((B, g * Hkv, 128), torch.bfloat16)
    la, lf = mk((B, g * Hkv), torch.float32), mk((B, g * Hkv), torch.float32)
    gen = synth.rng(92)
    for t in range(steps):
        k = H.dev_bf16(synth.normal_bf16(gen, (B, 1, Hkv, 128)))
        v = H.dev_bf16(synth.normal_bf16(gen, (B, 1, Hkv, 128)))
        q = H.dev_bf16(synth.normal_bf16(gen, (B, g * Hkv, 128)))
        resa.resa_commit_kv(A.struct, k, v, 1, False)
        resa.resa_select_blocks(A.struct, q, p, ia, ca, n_cap, wa, nb)
        resa.resa_sparse_decode(A.struct, q, ia, ca, n_cap, p, oa, la, 0, wa, nb)
        resa.resa_decode_step(F.struct, k, v, q, p, ifu, cf, n_cap, of, lf, 0, wf, nb)
        assert torch.equal(ia, ifu) and torch.equal(ca, cf), t
        assert np.array_equal(H.host_bits(oa), H.host_bits(of)), t
        assert np.array_equal(la.cpu().numpy().view(np.uint32), lf.cpu().numpy().view(np.uint32)), t
    assert resa.resa_read_device_error(A.struct) == (0, 0)
    assert resa.resa_read_device_error(F.struct) == (0, 0)
    assert torch.equal(A.seq_lens, F.seq_lens)
    assert A.seq_lens.cpu().tolist() == [T + steps for T in lens]
    assert np.array_equal(H.host_bits(A.k_pool), H.host_bits(F.k_pool))
    assert np.array_equal(H.host_bits(A.v_pool), H.host_bits(F.v_pool))
    sa, sf = H.host_bits(A.summaries), H.host_bits(F.summaries)
    for b, T in enumerate(lens):
        M = (T + steps + 15) // 16
        assert np.array_equal(sa[b, :, :M], sf[b, :, :M]), b


def test_decode_step_large_batch_equals_commit_select_decode():
    """Batch 40 at the 28/4 head geometry: 1,120 output rows, merged a row per
    warp, whose merge also advances seq_lens in the fused step. Ids, counts,
    outputs and log-sum-exps equal those of the three calls bit for bit, and
    every length grows by one per step."""
    B, Hkv, g, steps = 40, 4, 7, 3
    lens = [int(x) for x in synth.rng(96).integers(1, 400, size=B)]
    maxb = (max(lens) + steps + 15) // 16 + 2
    A, F = _decode_step_caches(lens, Hkv, g, maxb, 2, 97)
    p = resa.params(0.1, 4, 1)
    n_cap = resa.resa_max_selected(A.struct, p)
    wa, nb = H.workspace(A, n_cap)
    wf, _ = H.workspace(F, n_cap)
    mk = lambda shape, dt: torch.empty(shape, dtype=dt, device="cuda")
    ia, ifu = mk((B, Hkv, n_cap), torch.int32), mk((B, Hkv, n_cap), torch.int32)
    ca, cf = mk((B, Hkv), torch.int32), mk((B, Hkv), torch.int32)
    oa, of = mk((B, g * Hkv, 128), torch.bfloat16), mk((B, g * Hkv, 128), torch.bfloat16)
    la, lf = mk((B, g * Hkv), torch.float32), mk((B, g * Hkv), torch.float32)
    gen = synth.rng(98)
    for t in range(steps):
        k = H.dev_bf16(synth.normal_bf16(gen, (B, 1, Hkv, 128)))
        v = H.dev_bf16(synth.normal_bf16(gen, (B, 1, Hkv, 128)))
        q = H.dev_bf16(synth.normal_bf16(gen, (B, g * Hkv, 128)))
        resa.resa_commit_kv(A.struct, k, v, 1, False)
        resa.resa_select_blocks(A.struct, q, p, ia, ca, n_cap, wa, nb)
        resa.resa_sparse_decode(A.struct, q, ia, ca, n_cap, p, oa, la, 0, wa, nb)
        resa.resa_decode_step(F.struct, k, v, q, p, ifu, cf, n_cap, of, lf, 0, wf, nb)
        assert torch.equal(ia, ifu) and torch.equal(ca, cf), t
        assert np.array_equal(H.host_bits(oa), H.host_bits(of)), t
        assert np.array_equal(la.cpu().numpy().view(np.uint32), lf.cpu().numpy().view(np.uint32)), t
    assert resa.resa_read_device_error(A.struct) == (0, 0)
    assert resa.resa_read_device_error(F.struct) == (0, 0)
    assert A.seq_lens.cpu().tolist() == F.seq_lens.cpu().tolist() == [T + steps for T in lens]


def test_decode_step_sequence_at_capacity():
    """A sequence whose cache is full cannot take the appended token: the
    fused step reports RESA_DEV_SEQ_LEN_RANGE, gives it count 0 and ids -1,
    keeps its length, and serves the other sequences as the three calls do."""
    Hkv, g, maxb = 1, 4, 20
    lens = [300, maxb * 16]
    A, F = _decode_step_caches(lens, Hkv, g, maxb, 2, 93)
    p = resa.params(0.2, 2, 1)
    n_cap = resa.resa_max_selected(A.struct, p)
    wa, nb = H.workspace(A, n_cap)
    wf, _ = H.workspace(F, n_cap)
    gen = synth.rng(94)
    k = H.dev_bf16(synth.normal_bf16(gen, (2, 1, Hkv, 128)))
    v = H.dev_bf16(synth.normal_bf16(gen, (2, 1, Hkv, 128)))
    q = H.dev_bf16(synth.normal_bf16(gen, (2, g * Hkv, 128)))
    mk = lambda shape, dt: torch.empty(shape, dtype=dt, device="cuda")
    ia, ifu = mk((2, Hkv, n_cap), torch.int32), mk((2, Hkv, n_cap), torch.int32)
    ca, cf = mk((2, Hkv), torch.int32), mk((2, Hkv), torch.int32)
    oa, of = mk((2, g * Hkv, 128), torch.bfloat16), mk((2, g * Hkv, 128), torch.bfloat16)
    resa.resa_commit_kv(A.struct, k, v, 1, False)
    assert resa.resa_read_device_error(A.struct)[0] == 1
    resa.resa_select_blocks(A.struct, q, p, ia, ca, n_cap, wa, nb)
    resa.resa_sparse_decode(A.struct, q, ia, ca, n_cap, p, oa, None, 0, wa, nb)
    resa.resa_decode_step(F.struct, k, v, q, p, ifu, cf, n_cap, of, None, 0, wf, nb)
    code, detail = resa.resa_read_device_error(F.struct)
    assert (code, detail) == (1, 1)
    assert F.seq_lens.cpu().tolist() == [301, maxb * 16]
    assert cf[1].cpu().tolist() == [0] and np.all(ifu[1].cpu().numpy() == -1)
    assert torch.equal(ia[0], ifu[0]) and torch.equal(ca[0], cf[0])
    assert np.array_equal(H.host_bits(oa[0]), H.host_bits(of[0]))


# ------------------------------------------------------ Eq. 2 / Alg. 2 ----
def run_decode(cache, q_bits, sel_rows, n_cap, p, splits):
    """sel_rows[b][h] = block ids (any order)."""
    B, Hkv, Hq = cache.batch, cache.Hkv, cache.Hq
    idx = np.full((B, Hkv, n_cap), -1, dtype=np.int32)
    cnt = np.zeros((B, Hkv), dtype=np.int32)
    for b in range(B):
        for h in range(Hkv):
            s = np.asarray(sel_rows[b][h], dtype=np.int32)
            idx[b, h, :len(s)] = s
            cnt[b, h] = len(s)
    out = torch.empty((B, Hq, 128), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((B, Hq), dtype=torch.float32, device="cuda")
    ws, nb = H.workspace(cache, n_cap, splits)
    resa.resa_sparse_decode(cache.struct, H.dev_bf16(q_bits), torch.from_numpy(idx).cuda(),
                            torch.from_numpy(cnt).cuda(), n_cap, p, out, lse, splits, ws, nb)
    return H.host_f64(out), lse.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("g,Hkv,lens,nsel,splits", [
    (4, 2, [4100], 26, 0), (7, 4, [2053, 999], 40, 0), (7, 4, [2053, 999], 40, 1), (7, 4, [2053], 40, 7),
    (8, 1, [33], 3, 64), (1, 2, [500], 1, 0), (7, 1, [16 * 300 + 5], 300, 0), (2, 1, [17], 2, 3),
    (7, 2, [16 * 220 + 3], 200, 100),      # 100 splits: the merge takes two rounds of loads
    (5, 1, [3000], 100, 16), (3, 2, [1200, 700], 40, 0),
    (7, 4, [100 + 7 * i for i in range(37)], 6, 0),  # 1,036 output rows: the merge takes a warp per row
])
def test_sparse_decode_matches_oracle(g, Hkv, lens, nsel, splits):
    Ks, Vs = seq_inputs(10 + g, len(lens), Hkv, lens)
    maxb = max((T + 15) // 16 for T in lens) + 2
    cache = H.make_cache(Ks, Vs, g * Hkv, maxb)
    gr = synth.rng(77)
    q = synth.normal_bf16(gr, (len(lens), g * Hkv, 128))
    sel = []
    for b, T in enumerate(lens):
        M = (T + 15) // 16
        rows = []
        for h in range(Hkv):
            s = np.sort(gr.choice(M, size=min(nsel, M), replace=False))
            if M - 1 not in s:               # always include the partial last block
                s[-1] = M - 1
                s = np.unique(s)
            rows.append(s)
        sel.append(rows)
    n_cap = max(len(r) for rows in sel for r in rows) + 1
    p = resa.params(0.1, 0, 0)
    out, lse = run_decode(cache, q, sel, n_cap, p, splits)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    sc = 1 / math.sqrt(128)
    for b, T in enumerate(lens):
        Kf, Vf = O.widen_bf16(Ks[b]), O.widen_bf16(Vs[b])
        for h in range(Hkv):
            o, l = O.gbsa_attention(O.widen_bf16(q[b, h * g:(h + 1) * g]), Kf[h], Vf[h], T, sel[b][h], 16, sc)
            H.check_outputs(out[b, h * g:(h + 1) * g], o, f"b{b} h{h}")
            assert np.allclose(lse[b, h * g:(h + 1) * g], l, atol=2e-3, rtol=0)


def test_sparse_decode_all_blocks_equals_dense():
    g, Hkv, T = 7, 1, 16 * 64 - 3
    Ks, Vs = seq_inputs(21, 1, Hkv, [T])
    cache = H.make_cache(Ks, Vs, g, 64)
    q = synth.normal_bf16(synth.rng(22), (1, g, 128))
    out, _ = run_decode(cache, q, [[np.arange(64)]], 64, resa.params(1.0, 0, 0), 0)
    o, _ = O.dense_attention(O.widen_bf16(q[0]), O.widen_bf16(Ks[0][0]), O.widen_bf16(Vs[0][0]), T,
                             1 / math.sqrt(128))
    H.check_outputs(out[0], o, "dense")


def test_sparse_decode_empty_selection_gives_zero_and_neg_inf():
    Ks, Vs = seq_inputs(23, 1, 1, [64])
    cache = H.make_cache(Ks, Vs, 4, 4)
    q = synth.normal_bf16(synth.rng(24), (1, 4, 128))
    out, lse = run_decode(cache, q, [[np.zeros(0, dtype=np.int32)]], 4, resa.params(0.1, 0, 0), 0)
    assert np.all(out == 0) and np.all(np.isneginf(lse))


def test_sparse_decode_bad_block_id_is_reported_not_faulted():
    Ks, Vs = seq_inputs(25, 1, 1, [64])
    cache = H.make_cache(Ks, Vs, 4, 4)
    q = synth.normal_bf16(synth.rng(26), (1, 4, 128))
    out, _ = run_decode(cache, q, [[np.array([0, 7])]], 4, resa.params(0.1, 0, 0), 1)   # block 7 >= M = 4
    code, _ = resa.resa_read_device_error(cache.struct)
    assert code == 5
    o, _ = O.gbsa_attention(O.widen_bf16(q[0]), O.widen_bf16(Ks[0][0]), O.widen_bf16(Vs[0][0]), 64, [0], 16,
                            1 / math.sqrt(128))
    H.check_outputs(out[0], o, "bad id treated as masked")


# ------------------------------------------------------- rectification ----
@pytest.mark.parametrize("g,Hkv,lens,f", [
    (4, 2, [4100], 8), (7, 4, [2053, 640], 32), (7, 1, [1000], 16), (7, 1, [777], 64), (8, 2, [64], 64),
    (1, 1, [300], 8), (7, 2, [32], 32),
    (7, 4, [300, 280, 333, 290, 310, 305], 32),  # 5,376 rows of 5 splits: the merge takes a warp per row
])
def test_rectify_matches_oracle(g, Hkv, lens, f):
    Ks, Vs = seq_inputs(30 + f, len(lens), Hkv, lens)
    maxb = max((T + 15) // 16 for T in lens) + 2
    cache = H.make_cache(Ks, Vs, g * Hkv, maxb)
    gr = synth.rng(88)
    B = len(lens)
    qn = synth.normal_bf16(gr, (B, f, g * Hkv, 128))
    kn = synth.normal_bf16(gr, (B, f, Hkv, 128))
    vn = synth.normal_bf16(gr, (B, f, Hkv, 128))
    out = torch.empty((B, f, g * Hkv, 128), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((B, f, g * Hkv), dtype=torch.float32, device="cuda")
    ws, nb = H.workspace(cache, 8, 0, f)
    p = resa.params(0.1, 16, 1)
    resa.resa_rectify_attention(cache.struct, H.dev_bf16(qn), H.dev_bf16(kn), H.dev_bf16(vn), f, p, out, lse, ws, nb)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    out, lse = H.host_f64(out), lse.cpu().numpy()
    for b, T in enumerate(lens):
        o, l = O.rectify_attention(O.widen_bf16(qn[b]), O.widen_bf16(Ks[b]), O.widen_bf16(Vs[b]),
                                   O.widen_bf16(kn[b]), O.widen_bf16(vn[b]), T, 1 / math.sqrt(128))
        H.check_outputs(out[b], o, f"rectify b{b}")
        assert np.allclose(lse[b], l, atol=2e-3, rtol=0)


@pytest.mark.parametrize("L,C", [(1000, 256), (700, 700), (130, 64)])
def test_chunked_prefill_equals_dense_causal_attention(L, C):
    """Algorithm 1's prefill in chunks of C tokens: append the chunk's K/V to
    the cache (block keys built online), then the rectification call with
    f = C attends the chunk's queries causally to the cached prefix and the
    chunk itself. Every prompt position must match dense causal attention over
    the whole prompt, and the block keys the summaries of the whole prompt."""
    g, Hkv, B = 7, 2, 2
    gr = synth.rng(95 + C)
    Ks = [synth.normal_bf16(gr, (Hkv, L, 128)) for _ in range(B)]
    Vs = [synth.normal_bf16(gr, (Hkv, L, 128)) for _ in range(B)]
    Qs = [synth.normal_bf16(gr, (L, g * Hkv, 128)) for _ in range(B)]
    maxb = (L + 15) // 16 + 1
    empty = [np.zeros((Hkv, 0, 128), dtype=np.uint16)] * B
    cache = H.make_cache(empty, empty, g * Hkv, maxb)
    p = resa.params(0.1, 16, 1)
    ws, nb = H.workspace(cache, 8, 0, C)
    outs = []
    for c0 in range(0, L, C):
        f = min(C, L - c0)
        kc = np.stack([np.transpose(Ks[b][:, c0:c0 + f], (1, 0, 2)) for b in range(B)])   # [B, f, Hkv, d]
        vc = np.stack([np.transpose(Vs[b][:, c0:c0 + f], (1, 0, 2)) for b in range(B)])
        qc = np.stack([Qs[b][c0:c0 + f] for b in range(B)])                                 # [B, f, Hq, d]
        kd, vd = H.dev_bf16(kc), H.dev_bf16(vc)
        resa.resa_commit_kv(cache.struct, kd, vd, f, False)
        out = torch.empty((B, f, g * Hkv, 128), dtype=torch.bfloat16, device="cuda")
        resa.resa_rectify_attention(cache.struct, H.dev_bf16(qc), kd, vd, f, p, out, None, ws, nb)
        outs.append(H.host_f64(out))
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    assert cache.seq_lens.cpu().tolist() == [L] * B
    out = np.concatenate(outs, axis=1)
    summ = H.host_bits(cache.summaries)
    for b in range(B):
        K, V = O.widen_bf16(Ks[b]), O.widen_bf16(Vs[b])
        kall, vall = np.transpose(K, (1, 0, 2)), np.transpose(V, (1, 0, 2))
        o, _ = O.rectify_attention(O.widen_bf16(Qs[b]), K[:, :0], V[:, :0], kall, vall, L, 1 / math.sqrt(128))
        H.check_outputs(out[b], o, f"prefill b{b}")
        M = (L + 15) // 16
        for h in range(Hkv):
            kmin, kmax = O.block_summaries(K[h], 16)
            assert np.array_equal(O.widen_bf16(summ[b, h, :M, 0]), kmin)
            assert np.array_equal(O.widen_bf16(summ[b, h, :M, 1]), kmax)


@pytest.mark.parametrize("f", [16, 64])  # 384 output rows (a CTA per row) / 1,536 (a warp per row)
def test_active_mask_commit_and_rectify(f):
    """Continuous batching: only sequences with active[b] != 0 are rectified,
    appended to or overwritten; the others keep their cache, length, block
    keys and output rows, and record no error."""
    g, Hkv = 4, 2
    lens = [700, 333, 1025]
    B = len(lens)
    Ks, Vs = seq_inputs(97, B, Hkv, lens)
    maxb = max((T + 15) // 16 for T in lens) + 4
    cache = H.make_cache(Ks, Vs, g * Hkv, maxb)
    active = torch.tensor([1, 0, 1], dtype=torch.int32, device="cuda")
    gr = synth.rng(98)
    qn = synth.normal_bf16(gr, (B, f, g * Hkv, 128))
    kn = synth.normal_bf16(gr, (B, f, Hkv, 128))
    vn = synth.normal_bf16(gr, (B, f, Hkv, 128))
    p = resa.params(0.1, 16, 1)
    ws, nb = H.workspace(cache, 8, 0, f)
    out = torch.full((B, f, g * Hkv, 128), 7.0, dtype=torch.bfloat16, device="cuda")
    resa.resa_rectify_attention_active(cache.struct, active, H.dev_bf16(qn), H.dev_bf16(kn), H.dev_bf16(vn), f, p,
                                       out, None, ws, nb)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    o_host = H.host_f64(out)
    assert np.all(o_host[1] == 7.0)                      # left out: untouched
    for b in (0, 2):
        o, _ = O.rectify_attention(O.widen_bf16(qn[b]), O.widen_bf16(Ks[b]), O.widen_bf16(Vs[b]),
                                   O.widen_bf16(kn[b]), O.widen_bf16(vn[b]), lens[b], 1 / math.sqrt(128))
        H.check_outputs(o_host[b], o, f"rectify active b{b}")
    # overwrite commit of the f tokens: the left-out sequence keeps its K/V and block keys
    kp0, sm0 = H.host_bits(cache.k_pool).copy(), H.host_bits(cache.summaries).copy()
    resa.resa_commit_kv_active(cache.struct, active, H.dev_bf16(kn), H.dev_bf16(vn), f, True)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    sm1 = H.host_bits(cache.summaries)
    assert np.array_equal(sm1[1], sm0[1])
    for b in (0, 2):
        K, _ = H.logical_kv(cache, b)
        assert np.array_equal(np.transpose(K[:, lens[b] - f:], (1, 0, 2)), kn[b])
        kmin, kmax = O.block_summaries(O.widen_bf16(K[0]), 16)
        M = (lens[b] + 15) // 16
        assert np.array_equal(O.widen_bf16(sm1[b, 0, :M, 0]), kmin)
    K1, _ = H.logical_kv(cache, 1)
    assert np.array_equal(K1, Ks[1])
    # append of 3 tokens: only active sequences grow
    ka = synth.normal_bf16(gr, (B, 3, Hkv, 128))
    resa.resa_commit_kv_active(cache.struct, active, H.dev_bf16(ka), H.dev_bf16(ka), 3, False)
    assert cache.seq_lens.cpu().tolist() == [lens[0] + 3, lens[1], lens[2] + 3]
    assert resa.resa_read_device_error(cache.struct) == (0, 0)


@pytest.mark.parametrize("f,T", [(32, 3000), (16, 1500), (64, 1200)])
def test_rectify_rescale_path(f, T):
    """Keys whose magnitude ramps up along the positions (and log-normal
    outlier channels) make row maxima grow tile after tile, at different
    tiles for different rows, exercising the tensor-memory O rescale."""
    g, Hkv = 7, 2
    gr = synth.rng(90 + f)
    ramp = (1.0 + 6.0 * np.arange(T) / T)[None, :, None]
    chan = np.exp(0.7 * gr.standard_normal((Hkv, 1, 128)))
    Kf = gr.standard_normal((Hkv, T, 128)) * ramp * chan
    K = synth.f32_to_bf16_bits(Kf.astype(np.float32))
    V = synth.normal_bf16(gr, (Hkv, T, 128))
    cache = H.make_cache([K], [V], g * Hkv, (T + 15) // 16 + 2)
    qn = synth.normal_bf16(gr, (1, f, g * Hkv, 128))
    kn = np.ascontiguousarray(np.transpose(K[:, T - f:], (1, 0, 2)))[None]
    vn = np.ascontiguousarray(np.transpose(V[:, T - f:], (1, 0, 2)))[None]
    out = torch.empty((1, f, g * Hkv, 128), dtype=torch.bfloat16, device="cuda")
    ws, nb = H.workspace(cache, 8, 0, f)
    resa.resa_rectify_attention(cache.struct, H.dev_bf16(qn), H.dev_bf16(kn), H.dev_bf16(vn), f,
                                resa.params(0.1, 0, 0), out, None, ws, nb)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    o, _ = O.rectify_attention(O.widen_bf16(qn[0]), O.widen_bf16(K), O.widen_bf16(V), O.widen_bf16(kn[0]),
                               O.widen_bf16(vn[0]), T, 1 / math.sqrt(128))
    H.check_outputs(H.host_f64(out)[0], o, "rectify with growing maxima")


def test_rectify_too_short_sequence_is_reported():
    Ks, Vs = seq_inputs(40, 1, 1, [8])
    cache = H.make_cache(Ks, Vs, 4, 4)
    f = 16
    z = torch.zeros((1, f, 4, 128), dtype=torch.bfloat16, device="cuda")
    zk = torch.zeros((1, f, 1, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(z)
    ws, nb = H.workspace(cache, 4, 0, f)
    resa.resa_rectify_attention(cache.struct, z, zk, zk, f, resa.params(0.1, 0, 0), out, None, ws, nb)
    assert resa.resa_read_device_error(cache.struct)[0] == 1


def test_commit_beyond_capacity_is_reported_and_skipped():
    Ks, Vs = seq_inputs(41, 1, 1, [60])
    cache = H.make_cache(Ks, Vs, 2, 4)            # capacity 64
    kn = torch.zeros((1, 5, 1, 128), dtype=torch.bfloat16, device="cuda")
    resa.resa_commit_kv(cache.struct, kn, kn, 5, False)
    assert resa.resa_read_device_error(cache.struct)[0] == 1
    assert int(cache.seq_lens[0]) == 60


def test_bad_page_table_entry_is_reported():
    Ks, Vs = seq_inputs(42, 1, 1, [40])
    cache = H.make_cache(Ks, Vs, 2, 4)
    cache.page_table[0, 2] = 10 ** 6
    kn = torch.zeros((1, 1, 1, 128), dtype=torch.bfloat16, device="cuda")
    resa.resa_commit_kv(cache.struct, kn, kn, 1, False)
    assert resa.resa_read_device_error(cache.struct)[0] == 2
