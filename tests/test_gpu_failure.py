"""Failure detection and non-finite inputs on the GPU, with no fault and no hang.

* A bounded wait that runs out: the sparse decode kernel's copy-barrier poll
  limit is lowered to 0 through the C ABI, so every warp gives up at its
  first wait. The call must record RESA_DEV_WAIT_TIMEOUT, write zero outputs
  (nothing was attended) and leave the context usable: the next call with the
  default limit matches the oracle.
* NaN keys (the oracle's reading 10): a NaN makes its block's summary NaN in
  that dimension (bulk build and append commit alike), the block's score
  NaN, and the block ranks below every other in the top-n, so it is not
  selected while the budget allows and the decode output stays finite. A
  forced local block holding a NaN key is still selected; the output of its
  group is then NaN, as in the oracle.
"""
import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_04108_gb300 import resa, synth
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu

BF16_NAN = np.uint16(0x7FC0)
SCALE = 1 / math.sqrt(128)


def decode(cache, q_bits, sel_rows, n_cap, p):
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
    ws, nb = H.workspace(cache, n_cap, 0)
    resa.resa_sparse_decode(cache.struct, H.dev_bf16(q_bits), torch.from_numpy(idx).cuda(),
                            torch.from_numpy(cnt).cuda(), n_cap, p, out, lse, 0, ws, nb)
    return H.host_f64(out), lse.cpu().numpy().astype(np.float64)


def test_decode_wait_timeout_is_reported_then_recovers():
    g, Hkv, lens = 7, 2, [900, 1500]
    gr = synth.rng(7100)
    Ks = [synth.normal_bf16(gr, (Hkv, T, 128)) for T in lens]
    Vs = [synth.normal_bf16(gr, (Hkv, T, 128)) for T in lens]
    cache = H.make_cache(Ks, Vs, g * Hkv, max(lens) // 16 + 2)
    q = synth.normal_bf16(gr, (len(lens), g * Hkv, 128))
    sel = [[np.sort(gr.choice((T + 15) // 16, 24, replace=False)) for _ in range(Hkv)] for T in lens]
    p = resa.params(0.1, 0, 0)
    try:
        resa.resa_set_decode_wait_polls(0)
        out, lse = decode(cache, q, sel, 24, p)
        code, _ = resa.resa_read_device_error(cache.struct)
    finally:
        resa.resa_set_decode_wait_polls()
    assert code == 4, "RESA_DEV_WAIT_TIMEOUT expected"
    assert np.all(out == 0) and np.all(np.isneginf(lse))
    out, lse = decode(cache, q, sel, 24, p)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    for b, T in enumerate(lens):
        for h in range(Hkv):
            qg = O.widen_bf16(q[b, h * g:(h + 1) * g])
            o, l = O.gbsa_attention(qg, O.widen_bf16(Ks[b][h]), O.widen_bf16(Vs[b][h]), T, sel[b][h], 16, SCALE)
            H.check_outputs(out[b, h * g:(h + 1) * g], o, f"after timeout b{b} h{h}")
            assert np.allclose(lse[b, h * g:(h + 1) * g], l, atol=2e-3, rtol=0)


def test_nan_keys_rank_last_and_decode_stays_finite():
    g, Hkv, T = 7, 2, 2000
    M = (T + 15) // 16
    gr = synth.rng(7200)
    Ks = [synth.normal_bf16(gr, (Hkv, T, 128)) for _ in range(2)]
    Vs = [synth.normal_bf16(gr, (Hkv, T, 128)) for _ in range(2)]
    # sequence 0: NaN keys in three unforced blocks of head 0 and one of head 1
    for h, blk, row, dim in ((0, 3, 5, 17), (0, 10, 0, 100), (0, 50, 15, 0), (1, 77, 9, 64)):
        Ks[0][h, blk * 16 + row, dim] = BF16_NAN
    # sequence 1: a NaN key in the forced (last) block of head 1
    Ks[1][1, T - 3, 33] = BF16_NAN
    cache = H.make_cache(Ks, Vs, g * Hkv, M + 2)
    p = resa.params(0.1, 0, 1)
    n_cap = resa.resa_max_selected(cache.struct, p)
    # Eq. 3: summaries NaN exactly where the oracle's are
    summ = H.host_f64(cache.summaries)
    for b in range(2):
        for h in range(Hkv):
            mn, mx = O.block_summaries(O.widen_bf16(Ks[b][h]), 16)
            assert np.array_equal(summ[b, h, :M, 0], mn, equal_nan=True)
            assert np.array_equal(summ[b, h, :M, 1], mx, equal_nan=True)
    # Eq. 4 / 5 on the GPU
    q = synth.normal_bf16(gr, (2, g * Hkv, 128))
    idx = torch.empty((2, Hkv, n_cap), dtype=torch.int32, device="cuda")
    cnt = torch.empty((2, Hkv), dtype=torch.int32, device="cuda")
    ws, nb = H.workspace(cache, n_cap)
    resa.resa_select_blocks(cache.struct, H.dev_bf16(q), p, idx, cnt, n_cap, ws, nb)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    idx, cnt = idx.cpu().numpy(), cnt.cpu().numpy()
    sel = [[None] * Hkv for _ in range(2)]
    for b in range(2):
        for h in range(Hkv):
            mn, mx = O.block_summaries(O.widen_bf16(Ks[b][h]), 16)
            scores = O.quest_scores(O.pooled_query(O.widen_bf16(q[b, h * g:(h + 1) * g])), mn, mx)
            n = O.selection_budget(M, 0.1, 0, 1)
            assert cnt[b, h] == n
            sel[b][h] = idx[b, h, :n]
            H.check_selection(sel[b][h], scores, n, 1)
    nan_blocks = {(0, 0): {3, 10, 50}, (0, 1): {77}}
    for (b, h), blocks in nan_blocks.items():
        assert not blocks & set(sel[b][h].tolist()), "a NaN block was selected"
    assert M - 1 in sel[1][1].tolist()
    # Eq. 2: finite wherever the attended blocks are finite; NaN for the group with a NaN forced block
    out, _ = decode(cache, q, sel, n_cap, p)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    for b in range(2):
        for h in range(Hkv):
            qg = O.widen_bf16(q[b, h * g:(h + 1) * g])
            o, _ = O.gbsa_attention(qg, O.widen_bf16(Ks[b][h]), O.widen_bf16(Vs[b][h]), T, sel[b][h], 16, SCALE)
            got = out[b, h * g:(h + 1) * g]
            if (b, h) == (1, 1):
                assert np.isnan(o).all() and np.isnan(got).all()
            else:
                H.check_outputs(got, o, f"NaN keys unselected b{b} h{h}")


def test_nan_key_appended_poisons_its_block_summary():
    """The append commit folds a NaN key into its block's summary the same
    way the bulk build does (Eq. 3 online update, reading 10)."""
    Hkv, T = 2, 40
    gr = synth.rng(7300)
    K = synth.normal_bf16(gr, (Hkv, T, 128))
    V = synth.normal_bf16(gr, (Hkv, T, 128))
    cache = H.make_cache([K], [V], 4 * Hkv, 8)
    kn = synth.normal_bf16(gr, (1, 3, Hkv, 128))
    kn[0, 1, 0, 7] = BF16_NAN
    resa.resa_commit_kv(cache.struct, H.dev_bf16(kn), H.dev_bf16(kn), 3, False)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    Kall = np.concatenate([K, np.transpose(kn[0], (1, 0, 2))], axis=1)
    summ = H.host_f64(cache.summaries)
    M = (T + 3 + 15) // 16
    for h in range(Hkv):
        mn, mx = O.block_summaries(O.widen_bf16(Kall[h]), 16)
        assert np.array_equal(summ[0, h, :M, 0], mn, equal_nan=True)
        assert np.array_equal(summ[0, h, :M, 1], mx, equal_nan=True)
    assert np.isnan(summ[0, 0, 2, 0, 7]) and np.isnan(summ[0, 0, 2, 1, 7])


def test_nan_key_appended_by_the_fused_step():
    """The fused decode step folds the appended key into its block's summary
    inside the score kernel (Eq. 3 online update): a NaN key poisons that
    dimension there too, the block (the forced local one) is still selected,
    and the output of its group is NaN while the other group stays finite and
    matches the oracle."""
    g, Hkv, T = 4, 2, 300
    gr = synth.rng(7400)
    K = synth.normal_bf16(gr, (Hkv, T, 128))
    V = synth.normal_bf16(gr, (Hkv, T, 128))
    cache = H.make_cache([K], [V], g * Hkv, (T + 1 + 15) // 16 + 1)
    p = resa.params(0.1, 4, 1)
    n_cap = resa.resa_max_selected(cache.struct, p)
    kn = synth.normal_bf16(gr, (1, Hkv, 128))
    vn = synth.normal_bf16(gr, (1, Hkv, 128))
    kn[0, 1, 5] = BF16_NAN                       # KV head 1's appended key
    q = synth.normal_bf16(gr, (1, g * Hkv, 128))
    idx = torch.empty((1, Hkv, n_cap), dtype=torch.int32, device="cuda")
    cnt = torch.empty((1, Hkv), dtype=torch.int32, device="cuda")
    out = torch.empty((1, g * Hkv, 128), dtype=torch.bfloat16, device="cuda")
    ws, nb = H.workspace(cache, n_cap)
    resa.resa_decode_step(cache.struct, H.dev_bf16(kn), H.dev_bf16(vn), H.dev_bf16(q), p, idx, cnt, n_cap, out, None,
                          0, ws, nb)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    assert int(cache.seq_lens[0]) == T + 1
    Kall = np.concatenate([K, kn[0][:, None]], axis=1)
    Vall = np.concatenate([V, vn[0][:, None]], axis=1)
    summ = H.host_f64(cache.summaries)[0]
    M = (T + 1 + 15) // 16
    for h in range(Hkv):
        mn, mx = O.block_summaries(O.widen_bf16(Kall[h]), 16)
        assert np.array_equal(summ[h, :M, 0], mn, equal_nan=True)
        assert np.array_equal(summ[h, :M, 1], mx, equal_nan=True)
    idx, cnt, out = idx.cpu().numpy(), cnt.cpu().numpy(), H.host_f64(out)
    for h in range(Hkv):
        mn, mx = O.block_summaries(O.widen_bf16(Kall[h]), 16)
        qg = O.widen_bf16(q[0, h * g:(h + 1) * g])
        scores = O.quest_scores(O.pooled_query(qg), mn, mx)
        n = O.selection_budget(M, 0.1, 4, 1)
        sel = idx[0, h, :cnt[0, h]]
        H.check_selection(sel, scores, n, 1)
        assert M - 1 in sel.tolist()
        o, _ = O.gbsa_attention(qg, O.widen_bf16(Kall[h]), O.widen_bf16(Vall[h]), T + 1, sel, 16, SCALE)
        if h == 1:
            assert np.isnan(o).all() and np.isnan(out[0, h * g:(h + 1) * g]).all()
        else:
            H.check_outputs(out[0, h * g:(h + 1) * g], o, "fused step, finite group")
