"""Seeded synthetic inputs for the ReSA decode-attention path.

This module only draws random numbers and lays them out; it contains none of
the method's arithmetic (no summaries, scores, selection or attention). Both
the fp64 oracle and the CUDA path are fed from here, so that they see the
same bf16 bits.

Value recipes follow the paper's workloads (Qwen2.5-7B head geometry: 28
query heads, 4 KV heads, head dim 128, Section 3.2; block size 16, f = 32,
Section 3.1; contexts 16K-256K and batch 8, Section 3.5):

* Q, K, V ~ N(0, 1), rounded to bf16 (round to nearest even).
* Optional per-(KV head, channel) log-normal scale on K (outlier channels).
* "Sparse-era" keys/values are the dense ones plus 0.05 * N(0, 1): the error a
  sparse forward leaves in the cache, which rectification removes (Section 2.2).
* Optional needle blocks: a query is built as z + 2 * k_needle so that one
  block is strongly preferred (retrieval-shaped structure).

bf16 values are carried as uint16 bit patterns in numpy, and as
``torch.bfloat16`` tensors on the device.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass

import numpy as np

BLOCK_SIZE = 16
HEAD_DIM = 128
SPARSE_ERA_NOISE = 0.05


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> 16) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) >> 16
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32 (input plumbing only)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def normal_bf16(g: np.random.Generator, shape, scale: float = 1.0) -> np.ndarray:
    """N(0, scale^2) samples rounded to bf16, as uint16 bits."""
    x = g.standard_normal(size=shape, dtype=np.float32)
    if scale != 1.0:
        x *= np.float32(scale)
    return f32_to_bf16_bits(x)


def perturb_bf16(g: np.random.Generator, bits: np.ndarray, sigma: float = SPARSE_ERA_NOISE) -> np.ndarray:
    """bits + sigma * N(0, 1), re-rounded to bf16 (the sparse-era cache error)."""
    x = bf16_bits_to_f32(bits) + np.float32(sigma) * g.standard_normal(size=bits.shape, dtype=np.float32)
    return f32_to_bf16_bits(x)


def page_table(g: np.random.Generator, batch: int, max_blocks: int, num_pages: int | None = None) -> np.ndarray:
    """A random logical-block -> physical-page map with no page shared.

    Returns int32 [batch, max_blocks]; every entry is a distinct page id in
    [0, num_pages). Scattered pages make the paged gather honest.
    """
    total = batch * max_blocks
    if num_pages is None:
        num_pages = total
    if num_pages < total:
        raise ValueError("num_pages must cover batch * max_blocks")
    perm = g.permutation(num_pages)[:total].astype(np.int32)
    return perm.reshape(batch, max_blocks)


@dataclass(frozen=True)
class Workload:
    """One synthetic decode workload (sizes, ReSA parameters, value recipe)."""

    name: str
    batch: int
    num_q_heads: int
    num_kv_heads: int
    context: int            # tokens already in the cache when decoding starts
    steps: int              # decode steps
    f: int                  # rectification period (Algorithm 1)
    keep: float             # fraction of blocks attended (Eq. 5's ratio)
    n_min_blocks: int
    n_local_blocks: int
    seed: int
    head_dim: int = HEAD_DIM
    block_size: int = BLOCK_SIZE
    k_channel_sigma: float = 0.0   # log-normal sigma of per-channel K scale (0: none)
    layers: int = 1                # independent per-layer caches
    needle_blocks: int = 0         # per (sequence, KV head)

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    def capacity_tokens(self, extra_steps: int = 0) -> int:
        """Tokens the cache must hold: context + decode steps (+ slack), block aligned."""
        t = self.context + self.steps + extra_steps
        b = self.block_size
        return ((t + b - 1) // b) * b

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads of the hot path, named by what they are.
WORKLOADS = {
    # single layer, batch 1, 4K context, GQA 4 (8 q / 2 kv heads), keep 10%
    # (min 16 blocks = 256 tokens) + 4 local blocks (64 tokens), f = 8.
    "b1_h8kv2_ctx4k_f8": Workload(
        name="b1_h8kv2_ctx4k_f8", batch=1, num_q_heads=8, num_kv_heads=2, context=4096,
        steps=32, f=8, keep=0.10, n_min_blocks=16, n_local_blocks=4, seed=2506041081),
    # Qwen2.5-7B-shaped layer, batch 8, 32K context, sparsity 0.9, min 2048 tokens,
    # f = 32, log-normal per-channel K outliers.
    "qwen7b_b8_ctx32k_f32": Workload(
        name="qwen7b_b8_ctx32k_f32", batch=8, num_q_heads=28, num_kv_heads=4, context=32768,
        steps=64, f=32, keep=0.10, n_min_blocks=128, n_local_blocks=1, seed=2506041082,
        k_channel_sigma=1.0),
    # batch 4, 128K context, 28 independent per-layer caches, 256 steps, needles.
    "qwen7b_b4_ctx128k_28l_needles": Workload(
        name="qwen7b_b4_ctx128k_28l_needles", batch=4, num_q_heads=28, num_kv_heads=4,
        context=131072, steps=256, f=32, keep=0.10, n_min_blocks=128, n_local_blocks=1,
        seed=2506041083, layers=28, needle_blocks=16),
    # batch 1, 256K context, sparsity 0.95, min 2048 tokens, 512 steps.
    "qwen7b_b1_ctx256k_keep5": Workload(
        name="qwen7b_b1_ctx256k_keep5", batch=1, num_q_heads=28, num_kv_heads=4, context=262144,
        steps=512, f=32, keep=0.05, n_min_blocks=128, n_local_blocks=1, seed=2506041084),
}

# Latency breakdown (sparse step versus dense flash decoding of every block):
# the 32K batch-8 workload's geometry and ReSA parameters at these contexts.
BREAKDOWN_CONTEXTS = (16384, 65536, 262144)

# Chunked dense prefill: prompt lengths and chunk size.
PREFILL_LENGTHS = (32768, 131072)
PREFILL_CHUNK = 4096
PREFILL_SEED = 2506041086

# Rectification-only sweep: f new queries against cached contexts.
RECTIFY_SWEEP = [(t, f) for t in (16384, 65536, 262144) for f in (16, 32, 64)]
RECTIFY_SWEEP_SEED = 2506041085


@dataclass
class HostDecodeInputs:
    """Host-side (numpy, bf16 bits) inputs for one sequence batch.

    prefill_k / prefill_v : uint16 [B, Hkv, context, d]
    step_q                : uint16 [steps, B, Hq, d]
    step_k / step_v       : uint16 [steps, B, Hkv, d]   (sparse-era values)
    dense_k / dense_v     : uint16 [steps, B, Hkv, d]   (dense values written back
                            by rectification)
    dense_q               : uint16 [steps, B, Hq, d]    (queries of the dense re-encode)
    k_scale               : float32 [Hkv, d] per-channel K scale (ones if none)
    needles               : int32 [B, Hkv, needle_blocks] block ids (empty if none)
    """

    prefill_k: np.ndarray
    prefill_v: np.ndarray
    step_q: np.ndarray
    step_k: np.ndarray
    step_v: np.ndarray
    dense_q: np.ndarray
    dense_k: np.ndarray
    dense_v: np.ndarray
    k_scale: np.ndarray
    needles: np.ndarray


def channel_scale(g: np.random.Generator, num_kv_heads: int, head_dim: int, sigma: float) -> np.ndarray:
    if sigma <= 0.0:
        return np.ones((num_kv_heads, head_dim), dtype=np.float32)
    return np.exp(sigma * g.standard_normal((num_kv_heads, head_dim))).astype(np.float32)


def decode_inputs(w: Workload, context: int | None = None, steps: int | None = None,
                  batch: int | None = None, layer: int = 0) -> HostDecodeInputs:
    """Draw the host inputs of workload ``w`` (optionally at a reduced size).

    The stream is keyed on (seed, layer) so a reduced ``steps`` gives a prefix
    of a larger draw only for the prefill; tests always pass the sizes they use.
    """
    B = w.batch if batch is None else batch
    T0 = w.context if context is None else context
    S = w.steps if steps is None else steps
    Hq, Hkv, d = w.num_q_heads, w.num_kv_heads, w.head_dim
    g = rng(w.seed * 1000 + layer)
    scale = channel_scale(g, Hkv, d, w.k_channel_sigma)

    pk = g.standard_normal(size=(B, Hkv, T0, d), dtype=np.float32) * scale[None, :, None, :]
    prefill_k = f32_to_bf16_bits(pk)
    del pk
    prefill_v = normal_bf16(g, (B, Hkv, T0, d))
    dense_k = f32_to_bf16_bits(g.standard_normal(size=(S, B, Hkv, d), dtype=np.float32) * scale[None, None])
    dense_v = normal_bf16(g, (S, B, Hkv, d))
    step_k = perturb_bf16(g, dense_k)
    step_v = perturb_bf16(g, dense_v)
    dense_q = normal_bf16(g, (S, B, Hq, d))
    step_q = perturb_bf16(g, dense_q)

    needles = np.zeros((B, Hkv, 0), dtype=np.int32)
    if w.needle_blocks > 0:
        M0 = T0 // w.block_size
        needles = np.stack([np.stack([g.choice(M0, size=w.needle_blocks, replace=False)
                                      for _ in range(Hkv)]) for _ in range(B)]).astype(np.int32)
        gq = w.group
        pk_f = bf16_bits_to_f32(prefill_k)
        q = bf16_bits_to_f32(step_q).copy()
        for s in range(S):
            for b in range(B):
                for h in range(Hkv):
                    blk = needles[b, h, g.integers(w.needle_blocks)]
                    tok = blk * w.block_size + g.integers(w.block_size)
                    kstar = pk_f[b, h, tok]
                    z = g.standard_normal(size=(gq, d), dtype=np.float32)
                    q[s, b, h * gq:(h + 1) * gq] = z + 2.0 * kstar[None, :]
        step_q = f32_to_bf16_bits(q)
    return HostDecodeInputs(prefill_k, prefill_v, step_q, step_k, step_v,
                            dense_q, dense_k, dense_v, scale, needles)


def rectify_inputs(seed: int, batch: int, num_q_heads: int, num_kv_heads: int, context: int,
                   f: int, head_dim: int = HEAD_DIM):
    """Inputs of one rectification: cache of ``context`` tokens (the last f of
    them sparse-era), and the dense q/k/v of those f tokens.

    Returns (cache_k, cache_v [B, Hkv, context, d], q_new [B, f, Hq, d],
    k_new, v_new [B, f, Hkv, d]) as uint16 bf16 bits.
    """
    g = rng(seed)
    ck = normal_bf16(g, (batch, num_kv_heads, context, head_dim))
    cv = normal_bf16(g, (batch, num_kv_heads, context, head_dim))
    q_new = normal_bf16(g, (batch, f, num_q_heads, head_dim))
    k_new = np.ascontiguousarray(np.transpose(ck[:, :, context - f:], (0, 2, 1, 3)))
    v_new = np.ascontiguousarray(np.transpose(cv[:, :, context - f:], (0, 2, 1, 3)))
    # the cached tail holds the sparse-era (perturbed) version of the new tokens
    ck[:, :, context - f:] = perturb_bf16(g, ck[:, :, context - f:])
    cv[:, :, context - f:] = perturb_bf16(g, cv[:, :, context - f:])
    return ck, cv, q_new, k_new, v_new
