"""Helpers for the GPU parity tests: move seeded bf16 inputs into a paged
cache, read results back, and compare against the fp64 oracle with the
tolerances of the task (indices exact up to the near-tie rule; outputs
2e-2 max-abs and 1e-3 mean-abs)."""
from __future__ import annotations

import numpy as np
import torch

import oracle as O
from paper_2506_04108_gb300 import resa, synth

OUT_MAX_ABS = 2e-2
OUT_MEAN_ABS = 1e-3
GAP_REL = 1e-4


def dev_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def host_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def host_f64(t: torch.Tensor) -> np.ndarray:
    return O.widen_bf16(host_bits(t))


def make_cache(Ks, Vs, Hq, max_blocks, seed=1, zero_pools=False, compact=False, reserve_blocks=0):
    """Paged cache holding per-sequence keys/values Ks[b], Vs[b] (uint16 bits,
    [Hkv, T_b, d]; ragged T_b allowed), pages scattered by a seeded page table.
    Summaries are built with resa_update_summaries. `compact` gives pages only
    to the blocks the sequences hold plus `reserve_blocks` more each (the rest
    of each page-table row points at page 0): for wide page-table rows whose
    tail is never touched."""
    B = len(Ks)
    Hkv = Ks[0].shape[0]
    if compact:
        need = [min(max_blocks, (K.shape[1] + 15) // 16 + reserve_blocks) for K in Ks]
        perm = synth.rng(seed).permutation(max(1, sum(need))).astype(np.int32)
        pt = np.zeros((B, max_blocks), dtype=np.int32)
        off = 0
        for b, m in enumerate(need):
            pt[b, :m] = perm[off:off + m]
            off += m
    else:
        pt = synth.page_table(synth.rng(seed), B, max_blocks)
    cache = resa.PagedKVCache(B, Hq, Hkv, max_blocks, pt, zero_pools=zero_pools)
    kp = host_bits(cache.k_pool).copy()
    vp = host_bits(cache.v_pool).copy()
    lens = []
    for b in range(B):
        T = Ks[b].shape[1]
        t = np.arange(T)
        pages = pt[b, t // 16]
        kp[pages, :, t % 16, :] = np.transpose(Ks[b], (1, 0, 2))
        vp[pages, :, t % 16, :] = np.transpose(Vs[b], (1, 0, 2))
        lens.append(T)
    cache.k_pool.copy_(dev_bf16(kp))
    cache.v_pool.copy_(dev_bf16(vp))
    cache.seq_lens.copy_(torch.tensor(lens, dtype=torch.int32))
    resa.resa_update_summaries(cache.struct, 0, -1)
    return cache


def logical_kv(cache, b):
    """(K, V) bits [Hkv, T_b, d] of sequence b gathered from the pool."""
    T = int(cache.seq_lens[b])
    pt = cache.page_table[b].cpu().numpy()
    t = np.arange(T)
    kp = host_bits(cache.k_pool)
    vp = host_bits(cache.v_pool)
    K = np.transpose(kp[pt[t // 16], :, t % 16, :], (1, 0, 2))
    V = np.transpose(vp[pt[t // 16], :, t % 16, :], (1, 0, 2))
    return K, V


def oracle_state(Kb, Vb, capacity):
    """SequenceState for one sequence from bits [Hkv, T, d]."""
    Hkv, T, d = Kb.shape
    st = O.SequenceState(Hkv, capacity, d, 16)
    st.prefill(O.widen_bf16(Kb), O.widen_bf16(Vb))
    return st


def workspace(cache, n_cap, num_splits=0, max_f=0):
    nbytes = resa.resa_workspace_size(cache.struct, n_cap, num_splits, max_f)
    return torch.empty(nbytes, dtype=torch.uint8, device="cuda"), nbytes


def check_selection(gpu_sel, scores, n, n_local):
    """Selected ids must equal the oracle's top-n, except that where the
    oracle's score gap at the n-th boundary is below 1e-4 relative, blocks
    whose oracle score lies within that band of the boundary may differ.
    Returns True if the sets are identical."""
    gpu_sel = np.asarray(gpu_sel)
    M = len(scores)
    assert len(gpu_sel) == n, (len(gpu_sel), n)
    assert len(set(gpu_sel.tolist())) == n
    if n == 0:
        return True
    assert np.all(np.diff(gpu_sel) > 0), "indices must be ascending"
    assert gpu_sel.min() >= 0 and gpu_sel.max() < M
    want = O.select_blocks(scores, n, n_local)
    if np.array_equal(gpu_sel, want):
        return True
    eff = scores.astype(np.float64).copy()
    if n_local:
        eff[max(0, M - n_local):] = np.inf
    forced = set(range(max(0, M - n_local), M))
    assert forced <= set(gpu_sel.tolist()), "forced local blocks missing"
    s_sorted = np.sort(eff)[::-1]
    thr = s_sorted[n - 1]
    nxt = s_sorted[n] if n < M else -np.inf
    tol = GAP_REL * max(abs(thr), 1e-30)
    assert thr - nxt < tol, f"selection differs but boundary gap {(thr - nxt) / max(abs(thr), 1e-30):.3e} >= 1e-4"
    diff = set(gpu_sel.tolist()) ^ set(want.tolist())
    for i in diff:
        assert abs(eff[i] - thr) <= tol, f"block {i} (score {eff[i]}) outside the tie band of {thr}"
    return False


def round_bf16(x: np.ndarray) -> np.ndarray:
    """fp64 -> nearest bf16 (ties to even) -> fp64: the ABI's output format."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float64))
    return t.to(torch.bfloat16).to(torch.float64).numpy()


def check_outputs(gpu, ref, what=""):
    """GPU outputs are bf16 (the C ABI's output type); the oracle's are fp64.

    * max-abs <= 2e-2 against the unrounded fp64 result and against it
      rounded to bf16;
    * mean-abs <= 1e-3 against the fp64 result rounded to bf16 (the kernel's
      arithmetic error alone);
    * mean-abs against the unrounded fp64 result <= 1e-3 plus the mean error
      that rounding the exact result to bf16 itself leaves (ulp/4 on average:
      ~2e-3 for outputs of magnitude 1, ~1e-4 for the small outputs of long
      contexts): a bf16 output cannot do better than its own rounding.
    """
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert np.isfinite(gpu).all(), f"{what}: non-finite output"
    rounded = round_bf16(ref)
    raw = np.abs(gpu - ref)
    err = np.abs(gpu - rounded)
    floor = np.abs(rounded - ref).mean()
    assert raw.max() <= OUT_MAX_ABS, f"{what}: max-abs vs fp64 {raw.max():.3e} > {OUT_MAX_ABS}"
    assert err.max() <= OUT_MAX_ABS, f"{what}: max-abs {err.max():.3e} > {OUT_MAX_ABS}"
    assert err.mean() <= OUT_MEAN_ABS, f"{what}: mean-abs {err.mean():.3e} > {OUT_MEAN_ABS}"
    assert raw.mean() <= OUT_MEAN_ABS + floor, \
        f"{what}: mean-abs vs fp64 {raw.mean():.3e} > {OUT_MEAN_ABS} + bf16 rounding floor {floor:.3e}"
    return float(err.max()), float(err.mean())
