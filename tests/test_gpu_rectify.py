"""Rectification (Section 2.2; Algorithm 1 DenseForward) against the fp64
oracle at the sizes and launch shapes the kernel meets in use.

* The rectification sweep's own cells: f in {16, 32, 64} new tokens of the
  Qwen2.5-7B head geometry (28 query / 4 KV heads, batch 1) against cached
  contexts of 16K, 64K and 256K tokens, each followed by the overwrite commit
  and the refresh of the touched block keys. Every row of two of the four KV
  heads is compared with the oracle (all f tokens x 7 query heads), and the
  overwritten K/V and block keys bit for bit.
* A shape whose key splits each walk at least 16 prefix tiles, with keys
  whose magnitude ramps along the positions, so that in every CTA some query
  row's running maximum grows by more than 2^8 after the CTA's first tile:
  the test derives the CTAs' key ranges from resa_rectify_num_splits and
  checks that growth from the inputs before it compares the outputs, so the
  tensor-memory O rescale is known to run in every CTA.
"""
import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_04108_gb300 import resa, synth
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu

G, HKV, D = 7, 4, 128
SCALE = 1 / math.sqrt(D)
LOG2E = 1.4426950408889634
TILE = 64          # keys per rectification tile
RESCALE_LOG2 = 8.0  # the kernel rescales O when a row maximum grows by more than 2^8


def rectify(cache, qn, kn, vn, f):
    B = qn.shape[0]
    out = torch.empty((B, f, G * cache.Hkv, D), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((B, f, G * cache.Hkv), dtype=torch.float32, device="cuda")
    ws, nb = H.workspace(cache, 8, 0, f)
    resa.resa_rectify_attention(cache.struct, H.dev_bf16(qn), H.dev_bf16(kn), H.dev_bf16(vn), f,
                                resa.params(0.1, 16, 1), out, lse, ws, nb)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    return H.host_f64(out), lse.cpu().numpy()


def check_rows(out, lse, qn, Kb, Vb, kn, vn, T, heads, what):
    """Every (token, query head) row of the KV heads `heads` against
    oracle.rectify_attention on that head's group (out/lse of one sequence)."""
    for h in heads:
        sl = slice(h * G, (h + 1) * G)
        o, l = O.rectify_attention(O.widen_bf16(qn[:, sl]), O.widen_bf16(Kb[h:h + 1]), O.widen_bf16(Vb[h:h + 1]),
                                   O.widen_bf16(kn[:, h:h + 1]), O.widen_bf16(vn[:, h:h + 1]), T, SCALE)
        H.check_outputs(out[:, sl], o, f"{what} h{h}")
        assert np.allclose(lse[:, sl], l, atol=2e-3, rtol=0), f"{what} h{h}: lse"


@pytest.mark.parametrize("T", [16384, 65536, 262144])
def test_rectify_sweep_cells_match_oracle(T):
    """One cache per context; the f = 16, 32, 64 cells run in turn on it, each
    followed by its overwrite commit (the next cell's prefix includes the
    positions the previous one overwrote, and the host copy follows)."""
    gr = synth.rng(5000 + T // 1024)
    K = synth.normal_bf16(gr, (HKV, T, D))
    V = synth.normal_bf16(gr, (HKV, T, D))
    cache = H.make_cache([K], [V], G * HKV, (T + 15) // 16 + 1, seed=T)
    for f in (16, 32, 64):
        qn = synth.normal_bf16(gr, (1, f, G * HKV, D))
        kn = synth.normal_bf16(gr, (1, f, HKV, D))
        vn = synth.normal_bf16(gr, (1, f, HKV, D))
        out, lse = rectify(cache, qn, kn, vn, f)
        check_rows(out[0], lse[0], qn[0], K, V, kn[0], vn[0], T, (0, 3), f"T={T} f={f}")
        # overwrite commit of the f tokens; their K/V and the touched block keys, bit for bit
        resa.resa_commit_kv(cache.struct, H.dev_bf16(kn), H.dev_bf16(vn), f, True)
        assert resa.resa_read_device_error(cache.struct) == (0, 0)
        assert int(cache.seq_lens[0]) == T
        K[:, T - f:] = np.transpose(kn[0], (1, 0, 2))
        V[:, T - f:] = np.transpose(vn[0], (1, 0, 2))
        pt = cache.page_table[0].cpu().numpy()
        t = np.arange(T - f, T)
        kp, vp = H.host_bits(cache.k_pool), H.host_bits(cache.v_pool)
        assert np.array_equal(kp[pt[t // 16], :, t % 16, :], np.transpose(K[:, T - f:], (1, 0, 2)))
        assert np.array_equal(vp[pt[t // 16], :, t % 16, :], np.transpose(V[:, T - f:], (1, 0, 2)))
        b0, b1 = (T - f) // 16, (T - 1) // 16 + 1
        summ = H.host_f64(cache.summaries)[0]
        for h in range(HKV):
            kmin, kmax = O.block_summaries(O.widen_bf16(K[h, b0 * 16:T]), 16)
            assert np.array_equal(summ[h, b0:b1, 0], kmin) and np.array_equal(summ[h, b0:b1, 1], kmax)


def cta_ranges(T, f, splits):
    """Key ranges [k0, k1) of the prefix tiles of each split (the last split
    also attends to the f new tokens), as resa_rectify_num_splits states."""
    ntp = (T - f + TILE - 1) // TILE
    per = (ntp + splits - 1) // splits
    out = []
    for s in range(splits):
        t0, t1 = s * per, min(ntp, (s + 1) * per)
        out.append((t0 * TILE, min(T - f, t1 * TILE), s == splits - 1))
    return out, per


def test_rectify_rescale_branch_taken_in_every_cta():
    B, f, T = 8, 64, 64 * TILE + 64
    gr = synth.rng(6100)
    ramp = (1.0 + 12.0 * np.arange(T) / T)[None, :, None]
    Ks, Vs = [], []
    for _ in range(B):
        Ks.append(synth.f32_to_bf16_bits((gr.standard_normal((HKV, T, D)) * ramp).astype(np.float32)))
        Vs.append(synth.normal_bf16(gr, (HKV, T, D)))
    cache = H.make_cache(Ks, Vs, G * HKV, (T + 15) // 16 + 1, seed=61)
    qn = synth.normal_bf16(gr, (B, f, G * HKV, D))
    kn = np.stack([np.transpose(Ks[b][:, T - f:], (1, 0, 2)) for b in range(B)])
    vn = np.stack([np.transpose(Vs[b][:, T - f:], (1, 0, 2)) for b in range(B)])
    splits = resa.resa_rectify_num_splits(cache.struct, f)
    ranges, per = cta_ranges(T, f, splits)
    assert per >= 16, f"each CTA should walk >= 16 prefix tiles, got {per} ({splits} splits)"
    # rows of a row group: 256 rows = 32 tokens x 8 (padded) heads, rows of head j >= g never exist
    rows_per_group = 256
    for b in range(B):
        Kf = O.widen_bf16(Ks[b])
        for h in range(HKV):
            q = O.widen_bf16(qn[b, :, h * G:(h + 1) * G])                    # [f, g, d]
            logit = np.einsum("igd,td->igt", q, Kf[h]) * SCALE * LOG2E       # [f, g, T], log2 domain
            for rg in range((8 * f + rows_per_group - 1) // rows_per_group):
                toks = slice(rg * rows_per_group // 8, min(f, (rg + 1) * rows_per_group // 8))
                for s, (k0, k1, last) in enumerate(ranges):
                    # the CTA's tiles: its prefix tiles, then (last split) the tail tile of the new tokens
                    bounds = [(k, min(k + TILE, k1)) for k in range(k0, k1, TILE)]
                    if last:
                        bounds.append((T - f, T))
                    tile_max = []
                    for (a, e) in bounds:
                        lg = logit[toks, :, a:e]
                        if (a, e) == (T - f, T):       # causal mask of the new tokens: row i sees <= T - f + i
                            i = np.arange(toks.start, toks.stop)[:, None, None]
                            lg = np.where(np.arange(a, e)[None, None, :] <= T - f + i, lg, -np.inf)
                        tile_max.append(lg.max(axis=2))              # [tokens, g]
                    tile_max = np.stack(tile_max)                     # [tiles, tokens, g]
                    growth = tile_max[1:].max(axis=0) - tile_max[0]
                    assert growth.max() > RESCALE_LOG2 + 1.0, (b, h, rg, s, float(growth.max()))
    out = torch.empty((B, f, G * HKV, D), dtype=torch.bfloat16, device="cuda")
    lse = torch.empty((B, f, G * HKV), dtype=torch.float32, device="cuda")
    ws, nb = H.workspace(cache, 8, 0, f)
    resa.resa_rectify_attention(cache.struct, H.dev_bf16(qn), H.dev_bf16(kn), H.dev_bf16(vn), f,
                                resa.params(0.1, 0, 0), out, lse, ws, nb)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)
    out, lse = H.host_f64(out), lse.cpu().numpy()
    for b in range(B):
        check_rows(out[b], lse[b], qn[b], Ks[b], Vs[b], kn[b], vn[b], T, range(HKV), f"ramped b{b}")
