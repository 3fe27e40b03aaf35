#!/usr/bin/env python
"""Benchmark of the GB300 ReSA decode-attention path (one JSON line).

Workload (default ``qwen7b_b8_ctx32k_f32``): one attention layer of
Qwen2.5-7B geometry (28 query / 4 KV heads, head dim 128, bf16), batch 8,
32K-token context, block size 16, 10% of blocks kept (min 128 blocks, 1
forced local block), rectification every f = 32 steps, K with log-normal
per-channel outlier scales. Synthetic seeded data; no weights.

One benchmark STEP is one rectification period of the path (Algorithm 1):
f decode steps, each = commit the new token's K/V (+ summary update) ->
select blocks (Eq. 4/5) -> split-K sparse decode + combine (Algorithm 2),
then the dense rectification of those f tokens + overwrite commit. To keep
the HBM numbers honest the step runs over R independent layer caches in
rotation (the decode steps of one layer are separated by the other layers'
traffic, as in a model's layer loop); ``value`` is layer-tokens per second
(tokens pushed through one attention layer of the workload per second).

Timing: W warm-up steps, then K steps replayed from one CUDA graph per step,
timed with CUDA events on the replay stream between a barrier +
synchronize on both sides; max over ranks. Per-call durations for the
roofline come from one CUDA graph per call type holding the step's calls of
that type in step order, timed with CUDA events (total / calls).
"""
from __future__ import annotations

import argparse
import datetime
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2506_04108_gb300 import synth  # noqa: E402

METRIC = "decode attention tokens/s"
UNIT = "tokens/s"
DEFAULT_WORKLOAD = "qwen7b_b8_ctx32k_f32"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
HEAD_DIM = 128
BLOCK = 16


# ------------------------------------------------------------ algorithmic work
def budget(M: int, keep: float, n_min: int, n_local: int) -> int:
    return min(M, max(n_min, math.ceil(M * keep), n_local))


def decode_bytes(B, Hq, Hkv, T, keep, n_min, n_local) -> int:
    """Bytes one sparse-decode call must move: K+V of the attended tokens
    (selected blocks, the partial last block counted by its valid tokens),
    the queries in and the outputs out."""
    M = (T + BLOCK - 1) // BLOCK
    n = budget(M, keep, n_min, n_local)
    tokens = (n - 1) * BLOCK + (T - BLOCK * (M - 1))
    return B * Hkv * tokens * 2 * HEAD_DIM * 2 + 2 * B * Hq * HEAD_DIM * 2


def select_bytes(B, Hq, Hkv, T, keep, n_min, n_local) -> int:
    """Summaries read (Eq. 4 reads k_min and k_max of every block), fp32 scores
    written and read back, queries read, indices written."""
    M = (T + BLOCK - 1) // BLOCK
    n = budget(M, keep, n_min, n_local)
    return B * Hkv * M * 2 * HEAD_DIM * 2 + B * Hkv * M * 8 + B * Hq * HEAD_DIM * 2 + B * Hkv * n * 4


def commit_bytes(B, Hkv, n_tokens) -> int:
    """New K/V read and written, plus one summary read+write per touched block."""
    return B * Hkv * n_tokens * HEAD_DIM * 2 * 2 * 2 + B * Hkv * 2 * (2 * HEAD_DIM * 2)


def rectify_bytes(B, Hq, Hkv, T, f) -> int:
    """K+V of all T positions per (sequence, KV head), queries in, outputs out."""
    return B * Hkv * T * 2 * HEAD_DIM * 2 + 2 * B * f * Hq * HEAD_DIM * 2


def rectify_flops(B, Hq, T, f) -> int:
    """Useful causal pairs only: 4 * d flops per (query head, visible key)."""
    return 4 * HEAD_DIM * Hq * B * (f * T - f * (f - 1) // 2)


def eq6_ratio(b: int, keep: float, f: int) -> float:
    """Eq. 6's memory ratio of the step relative to dense decoding."""
    return 1.0 / b + keep + 1.0 / f


# ------------------------------------------------------------------ helpers
def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as fh:
            return json.load(fh), "measured"
    return FALLBACK_PEAKS, "fallback"


def source_hash(*names) -> str:
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2506_04108_gb300", "csrc", n), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(call: str, workload: str, src_hash: str):
    """DRAM bytes per call of type `call` (summed over the call's kernels) from
    a committed ncu summary, if its recorded source hash still matches the
    kernel source; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as fh:
        table = json.load(fh)
    e = table.get(call, {}).get(workload)
    if not e or e.get("source_hash") != src_hash:
        return None
    return e.get("dram_bytes_per_call")


class ClockSampler:
    """nvidia-smi clock / throttle sampling every 20 ms. Between begin() and
    end() (host times bracketing a synchronised timed region) only the
    samples taken inside that window are summarised; without a window, or if
    none fell inside it, all of them are, and the summary says which."""

    QUERY = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu_index = gpu_index
        self.proc = None
        self.path = None
        self.window = None

    def begin(self):
        self.window = [datetime.datetime.now(), None]

    def end(self):
        if self.window is not None:
            self.window[1] = datetime.datetime.now()

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="resa_clocks_", suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu_index), f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "20"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None or self.path is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        rows = []
        with open(self.path) as fh:
            for line in fh:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 10:
                    continue
                try:
                    t = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f")
                    rows.append((t, float(parts[2]), float(parts[3]),
                                 {nm for nm, v in zip(names, parts[6:10]) if v.lower() == "active"}))
                except ValueError:
                    continue
        os.unlink(self.path)
        scope = "all samples"
        if self.window is not None and self.window[1] is not None:
            inside = [r for r in rows if self.window[0] <= r[0] <= self.window[1]]
            if inside:
                rows, scope = inside, "timed region"
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(r[1] for r in rows), "sm_max_mhz": max(r[2] for r in rows),
                "reasons": sorted(set().union(*(r[3] for r in rows))), "samples": len(rows), "window": scope}


# --------------------------------------------------------------- distributed
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def init_dist(backend: str):
    import torch.distributed as dist
    rank, world, _ = dist_env()
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend, rank=rank, world_size=world)
    return rank, world


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


def max_over_ranks(x: float, device=None) -> float:
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(units_per_rank: float, seconds_max: float, world: int) -> float:
    """Whole-job throughput: units processed by all ranks / the slowest rank's time."""
    return units_per_rank * world / seconds_max


# ---------------------------------------------------------------- GPU side
class LayerCache:
    """One layer's paged cache plus the device inputs/outputs of one period."""

    def __init__(self, w: synth.Workload, capacity_tokens: int, seed: int, device):
        import torch
        from paper_2506_04108_gb300 import resa
        self.w, self.resa = w, resa
        B, Hq, Hkv, f = w.batch, w.num_q_heads, w.num_kv_heads, w.f
        maxb = capacity_tokens // BLOCK
        gen = synth.rng(seed)
        pt = synth.page_table(gen, B, maxb)
        self.cache = resa.PagedKVCache(B, Hq, Hkv, maxb, pt, device=device, zero_pools=False)
        tg = torch.Generator(device=device)
        tg.manual_seed(seed)
        scale = torch.from_numpy(synth.channel_scale(gen, Hkv, HEAD_DIM, w.k_channel_sigma)).to(device)
        for pool, sc in ((self.cache.k_pool, scale), (self.cache.v_pool, None)):
            for i in range(0, pool.shape[0], 4096):            # fill in chunks to bound temporaries
                x = torch.randn(pool[i:i + 4096].shape, generator=tg, device=device)
                if sc is not None:
                    x *= sc[None, :, None, :]
                pool[i:i + 4096].copy_(x)
        self.cache.seq_lens.fill_(w.context)
        resa.resa_update_summaries(self.cache.struct, 0, -1)
        self.p = resa.params(w.keep, w.n_min_blocks, w.n_local_blocks)
        self.n_cap = resa.resa_max_selected(self.cache.struct, self.p)
        self.ws_bytes = resa.resa_workspace_size(self.cache.struct, self.n_cap, 0, f)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        self.idx = torch.empty((B, Hkv, self.n_cap), dtype=torch.int32, device=device)
        self.cnt = torch.empty((B, Hkv), dtype=torch.int32, device=device)

        def rn(*shape, s=1.0):
            return (torch.randn(shape, generator=tg, device=device) * s).to(torch.bfloat16)
        dk = rn(f, B, Hkv, HEAD_DIM) * scale[None, None].to(torch.bfloat16)
        dv = rn(f, B, Hkv, HEAD_DIM)
        dq = rn(f, B, Hq, HEAD_DIM)
        noise = synth.SPARSE_ERA_NOISE
        # per-step inputs of the sparse decode steps (sparse-era K/V and queries)
        self.q = (dq.float() + noise * torch.randn(dq.shape, generator=tg, device=device)).to(torch.bfloat16)
        self.k = (dk.float() + noise * torch.randn(dk.shape, generator=tg, device=device)).to(torch.bfloat16)
        self.v = (dv.float() + noise * torch.randn(dv.shape, generator=tg, device=device)).to(torch.bfloat16)
        # dense re-encode of the f tokens, [B, f, H, d]
        self.rq = dq.transpose(0, 1).contiguous()
        self.rk = dk.transpose(0, 1).contiguous()
        self.rv = dv.transpose(0, 1).contiguous()
        self.out = torch.empty((f, B, Hq, HEAD_DIM), dtype=torch.bfloat16, device=device)
        self.rout = torch.empty((B, f, Hq, HEAD_DIM), dtype=torch.bfloat16, device=device)
        self.needle_target = None
        if w.needle_blocks > 0:
            # Needle workload: per (sequence, KV head) a seeded set of needle
            # blocks of the prompt; at each step every query head of the group
            # is q = z + 2 k*, k* a random key of a random needle block (the
            # recipe of synth.decode_inputs, drawn here on the device pools).
            gn = synth.rng(seed * 7 + 3)
            g, nb = w.group, w.needle_blocks
            needles = np.stack([np.stack([gn.choice(w.context // BLOCK, size=nb, replace=False)
                                          for _ in range(Hkv)]) for _ in range(B)])          # [B, Hkv, nb]
            pick = gn.integers(nb, size=(f, B, Hkv))
            row = gn.integers(BLOCK, size=(f, B, Hkv))
            blk = np.take_along_axis(np.broadcast_to(needles, (f, B, Hkv, nb)), pick[..., None], axis=3)[..., 0]
            page = pt[np.arange(B)[None, :, None], blk]
            heads = np.broadcast_to(np.arange(Hkv)[None, None, :], blk.shape)
            kstar = self.cache.k_pool[torch.from_numpy(page).long().to(device),
                                      torch.from_numpy(np.ascontiguousarray(heads)).long().to(device),
                                      torch.from_numpy(row).long().to(device)].float()       # [f, B, Hkv, d]
            z = torch.randn((f, B, Hkv, g, HEAD_DIM), generator=tg, device=device)
            self.q = (z + 2.0 * kstar[:, :, :, None, :]).reshape(f, B, Hq, HEAD_DIM).to(torch.bfloat16)
            self.needle_target = torch.from_numpy(blk.astype(np.int32)).to(device)              # [f, B, Hkv]

    # kernels per call: the fused decode step 4 (score, top-n, decode, merge),
    # rectify 2, overwrite 1
    KERNELS_PER_DECODE_STEP = 4
    KERNELS_PER_RECTIFY = 3

    def commit(self, t):
        self.resa.resa_commit_kv(self.cache.struct, self.k[t], self.v[t], 1, False)

    def select(self, t):
        self.resa.resa_select_blocks(self.cache.struct, self.q[t], self.p, self.idx, self.cnt, self.n_cap, self.ws,
                                     self.ws_bytes)

    def sparse_decode(self, t):
        self.resa.resa_sparse_decode(self.cache.struct, self.q[t], self.idx, self.cnt, self.n_cap, self.p,
                                     self.out[t], None, 0, self.ws, self.ws_bytes)

    def rectify_attention(self):
        self.resa.resa_rectify_attention(self.cache.struct, self.rq, self.rk, self.rv, self.w.f, self.p,
                                         self.rout, None, self.ws, self.ws_bytes)

    def overwrite(self):
        self.resa.resa_commit_kv(self.cache.struct, self.rk, self.rv, self.w.f, True)

    def decode(self, t):
        """One decode step of Algorithm 1 for this layer: the fused call that
        appends the token, selects and decodes (= commit + select + decode)."""
        self.resa.resa_decode_step(self.cache.struct, self.k[t], self.v[t], self.q[t], self.p, self.idx, self.cnt,
                                   self.n_cap, self.out[t], None, 0, self.ws, self.ws_bytes)

    def rectify(self):
        """Rectification branch of Algorithm 1 for this layer."""
        self.rectify_attention()
        self.overwrite()


def needle_recall(layers) -> dict:
    """Informational: the fraction of (step, sequence, KV head) where the
    needle block the query was built from is among the selected blocks, over
    one eager period of fused decode steps on every layer (not timed)."""
    import torch
    f = layers[0].w.f
    hits = torch.zeros((), dtype=torch.int64, device=layers[0].idx.device)
    n = 0
    for t in range(f):
        for Lc in layers:
            Lc.decode(t)
            hits += (Lc.idx == Lc.needle_target[t][..., None]).any(dim=-1).sum()
            n += Lc.needle_target[t].numel()
    check_device_errors(layers)
    return {"value": round(int(hits.item()) / n, 4), "samples": n, "informational": True,
            "what": "needle block of the step's query selected (Eq. 4/5), one period on every layer"}


def run_period(layers):
    f = layers[0].w.f
    for t in range(f):
        for L in layers:
            L.decode(t)
    for L in layers:
        L.rectify()


def host_logical_kv(cache, b: int, T: int):
    """K, V bits [Hkv, T, d] of sequence b gathered from the device pool."""
    import torch
    pt = cache.page_table[b].cpu().numpy()
    t = np.arange(T)
    pages = torch.from_numpy(pt[t // BLOCK]).long().to(cache.k_pool.device)
    rows = torch.from_numpy(t % BLOCK).long().to(cache.k_pool.device)
    K = cache.k_pool[pages, :, rows, :].transpose(0, 1).contiguous()
    V = cache.v_pool[pages, :, rows, :].transpose(0, 1).contiguous()
    to_bits = lambda x: x.cpu().view(torch.int16).numpy().view(np.uint16)  # noqa: E731
    return to_bits(K), to_bits(V)


def bits(t):
    import torch
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


# ------------------------------------------------------------ oracle sample
def oracle_period(sample: dict) -> float:
    """One rectification period of the fp64 oracle for one sequence of one
    layer (f decode steps + rectification); returns the seconds it took.
    The state's prefill summaries are built before the clock starts."""
    import oracle as O
    K, V = O.widen_bf16(sample["K"]), O.widen_bf16(sample["V"])
    Hkv, T0, d = K.shape
    f = int(sample["f"])
    st = O.SequenceState(Hkv, T0 + f + BLOCK, d, BLOCK)
    st.prefill(K, V)
    p = O.ResaParams(float(sample["keep"]), int(sample["n_min"]), int(sample["n_local"]))
    q, k, v = (O.widen_bf16(sample[x]) for x in ("q", "k", "v"))
    rq, rk, rv = (O.widen_bf16(sample[x]) for x in ("rq", "rk", "rv"))
    t0 = time.perf_counter()
    for i in range(f):
        O.sparse_decode_step(st, q[i], k[i], v[i], p)
    O.rectify_step(st, rq, rk, rv, p)
    return time.perf_counter() - t0


def run_oracle_subprocess(sample: dict, threads: int = 1, repeats: int = 1, min_seconds: float = 0.0):
    """Time oracle_period `repeats` times, then more until `min_seconds` of
    work have been timed (at most ORACLE_MAX_REPEATS periods), in a fresh
    process whose BLAS/OpenMP pools are pinned to `threads` (so `cores` is
    what the oracle actually used); returns the list of per-repeat seconds."""
    with tempfile.TemporaryDirectory() as d:
        path = os.path.join(d, "sample.npz")
        np.savez(path, **sample)
        env = dict(os.environ)
        for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
            env[v] = str(threads)
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-worker", path,
                            "--repeats", str(repeats), "--min-seconds", str(min_seconds)],
                           env=env, capture_output=True, text=True, timeout=3600)
        if r.returncode != 0:
            raise RuntimeError(f"oracle worker failed: {r.stderr[-2000:]}")
        return json.loads(r.stdout.strip().splitlines()[-1])["seconds"]


def host_sample(w: synth.Workload, context: int):
    """The oracle's input sample drawn on the host with the workload's recipe:
    one sequence of one layer at the workload's context, one period of inputs."""
    inp = synth.decode_inputs(w, context=context, steps=w.f, batch=1)
    return {"K": inp.prefill_k[0], "V": inp.prefill_v[0], "q": inp.step_q[:, 0], "k": inp.step_k[:, 0],
            "v": inp.step_v[:, 0], "rq": inp.dense_q[:, 0], "rk": inp.dense_k[:, 0], "rv": inp.dense_v[:, 0],
            "f": w.f, "keep": w.keep, "n_min": w.n_min_blocks, "n_local": w.n_local_blocks}


# ------------------------------------------------------------------- arms
def run_reference(args, w: synth.Workload):
    """The oracle as it stands, timed on the host cores: each step is one
    period of one sequence of one layer (a bounded sample of the workload)."""
    rank, world, _ = dist_env()
    if world > 1 and rank != 0:
        return
    sample = host_sample(w, w.context)
    times = run_oracle_subprocess(sample, threads=1, repeats=args.warmup + args.steps)
    per_step = times[args.warmup:]
    tot = sum(per_step)
    value = args.steps * w.f / tot
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_of(w, args),
            "cpu_baseline": {"kind": "oracle", "value": value, "unit": UNIT, "cores": 1,
                             "sample": f"per step: 1 of {w.batch} sequences, 1 layer, {w.f} decode steps + "
                                       f"1 rectification at context {w.context} (fp64 numpy, 1 BLAS thread)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def config_of(w: synth.Workload, args) -> dict:
    return {"workload": w.name, "batch": w.batch, "context": w.context, "q_heads": w.num_q_heads,
            "kv_heads": w.num_kv_heads, "head_dim": HEAD_DIM, "block_size": BLOCK, "keep": w.keep,
            "n_min_blocks": w.n_min_blocks, "n_local_blocks": w.n_local_blocks, "f": w.f,
            "layers_rotated": args.layers,
            "step": f"{w.f} decode steps (resa_decode_step: append + select + decode) + 1 rectification "
                    f"(resa_rectify_attention + overwrite commit) per layer",
            "l2": f"{args.layers} independent layer caches rotated per decode step (other layers' traffic "
                  f"between reuses exceeds the 129 MB L2)", "parallelism": f"replicas x{args.gpus} (weak)"}


def capture(fn, device):
    """CUDA graph of the C-ABI calls `fn` issues (captured on a side stream)."""
    import torch
    stream = torch.cuda.Stream(device=device)
    stream.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        fn()
    torch.cuda.synchronize()
    return graph


def time_graph(graph, reps: int) -> float:
    """Mean seconds of one replay, CUDA events on the replay stream."""
    import torch
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        graph.replay()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / 1e3 / reps


def check_device_errors(layers):
    from paper_2506_04108_gb300 import resa
    for Lc in layers:
        code, detail = resa.resa_read_device_error(Lc.cache.struct)
        if code:
            raise RuntimeError(f"device error {resa.DEVICE_ERRORS.get(code)} detail {detail}")


# The step is decode_step (f x L), rectify and overwrite (L each); select,
# decode and commit are the pieces decode_step fuses, timed as their own calls
# for the per-kernel rooflines. decode_step and commit append f tokens per
# replay of their graph.
IN_STEP = ("decode_step", "rectify", "overwrite")
APPENDING_KINDS = ("decode_step", "commit")


def time_call_kinds(layers, device):
    """Mean microseconds per call of each call type: one CUDA graph per type
    holding the period's calls of that type in step order (f x L or L calls),
    one warm replay, then ATTR_REPS replays timed with CUDA events. The two
    appending types advance every sequence by f * (1 + ATTR_REPS) tokens."""
    f, L = layers[0].w.f, len(layers)
    kinds = {
        "decode_step": lambda: [Lc.decode(t) for t in range(f) for Lc in layers],
        "select": lambda: [Lc.select(t) for t in range(f) for Lc in layers],
        "decode": lambda: [Lc.sparse_decode(t) for t in range(f) for Lc in layers],
        "rectify": lambda: [Lc.rectify_attention() for Lc in layers],
        "overwrite": lambda: [Lc.overwrite() for Lc in layers],
        "commit": lambda: [Lc.commit(t) for t in range(f) for Lc in layers],
    }
    ncalls = {"decode_step": f * L, "select": f * L, "decode": f * L, "rectify": L, "overwrite": L, "commit": f * L}
    mean_us = {}
    for kind, fn in kinds.items():
        gk = capture(fn, device)             # capture does not execute
        gk.replay()                          # warm
        mean_us[kind] = time_graph(gk, ATTR_REPS) / ncalls[kind] * 1e6
        del gk
    check_device_errors(layers)
    return mean_us, ncalls


def call_bytes(w: synth.Workload, T: int) -> dict:
    """Algorithmic bytes of one call of each type at context T (select at the
    middle of the appending replays' range)."""
    B, f = w.batch, w.f
    Tm = T + f // 2
    return {
        "decode_step": (commit_bytes(B, w.num_kv_heads, 1) +
                        select_bytes(B, w.num_q_heads, w.num_kv_heads, Tm, w.keep, w.n_min_blocks, w.n_local_blocks) +
                        decode_bytes(B, w.num_q_heads, w.num_kv_heads, T, w.keep, w.n_min_blocks,
                                     w.n_local_blocks)),
        "commit": commit_bytes(B, w.num_kv_heads, 1),
        "select": select_bytes(B, w.num_q_heads, w.num_kv_heads, Tm, w.keep, w.n_min_blocks, w.n_local_blocks),
        "decode": decode_bytes(B, w.num_q_heads, w.num_kv_heads, T, w.keep, w.n_min_blocks, w.n_local_blocks),
        "rectify": rectify_bytes(B, w.num_q_heads, w.num_kv_heads, T, f),
        "overwrite": commit_bytes(B, w.num_kv_heads, f),
    }


def run_ours(args, w: synth.Workload):
    import torch
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    if world > 1:
        init_dist("nccl")
    from paper_2506_04108_gb300 import build as _b
    from paper_2506_04108_gb300 import resa
    _b.build()
    resa.load()

    if args.layers is None:
        args.layers = max(4, w.layers)
    L, f, B = args.layers, w.f, w.batch
    # periods that append f tokens: warm-up call, graph warm-up/timed/e2e replays, attribution commits
    periods_total = 1 + args.warmup + args.steps + (2 + args.steps) + 2 * (1 + ATTR_REPS) + 1
    capacity = ((w.context + f * periods_total + BLOCK) // BLOCK + 1) * BLOCK
    layers = [LayerCache(w, capacity, w.seed * 100 + 17 * rank + i, device) for i in range(L)]
    torch.cuda.synchronize()
    T = w.context                           # tokens in every sequence of every layer

    # warm-up call outside any graph (sets kernel attributes), then capture one step
    run_period(layers)
    T += f
    graph = capture(lambda: run_period(layers), device)
    for _ in range(args.warmup):
        graph.replay()
        T += f
    torch.cuda.synchronize()
    check_device_errors(layers)

    # ---- timed region ----
    T_timed0 = T
    with ClockSampler(local) as clocks:
        barrier()
        torch.cuda.synchronize()
        clocks.begin()
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record()
        for _ in range(args.steps):
            graph.replay()
        s1.record()
        torch.cuda.synchronize()
        clocks.end()
        barrier()
    T += f * args.steps
    secs = s0.elapsed_time(s1) / 1e3
    secs_max = max_over_ranks(secs, device)
    tokens_per_rank = B * f * L * args.steps
    value = aggregate(tokens_per_rank, secs_max, world)
    clk = clocks.summary()

    # ---- end to end through the public API with host buffers ----
    e2e = run_e2e(args, layers)
    T += f * (args.steps + 2)  # the timed steps and one warm replay of each buffer set's graph

    # ---- per-call durations: one graph per call type, the period's calls of that type in order ----
    T_attr = T
    mean_us, ncalls = time_call_kinds(layers, device)
    T += f * 2 * (1 + ATTR_REPS)
    in_step = IN_STEP
    algo = call_bytes(w, T_attr)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    per_step_us = {k: mean_us[k] * ncalls[k] for k in mean_us}
    tot = sum(per_step_us[k] for k in in_step)
    calls = {}
    for k in mean_us:
        gbs = algo[k] / (mean_us[k] * 1e-6) / 1e9
        calls[k] = {"us_per_call": round(mean_us[k], 2), "calls_per_step": ncalls[k], "GB/s": round(gbs, 1),
                    "frac_hbm": round(gbs / hbm, 3), "algorithmic_bytes": int(algo[k])}
        if k in in_step:
            calls[k]["share_of_step"] = round(per_step_us[k] / tot, 3)
        else:
            calls[k]["part_of"] = "decode_step"
            calls[k]["share_of_decode_step"] = round(mean_us[k] / mean_us["decode_step"], 3)
    rflops = rectify_flops(B, w.num_q_heads, T_attr, f)
    calls["rectify"]["TFLOP/s"] = round(rflops / (mean_us["rectify"] * 1e-6) / 1e12, 1)
    calls["rectify"]["frac_bf16_sustained"] = round(rflops / (mean_us["rectify"] * 1e-6) / 1e12 /
                                                    float(peaks["bf16_tflops_sustained"]), 3)
    # dominant kernel pair: the largest per-step time among the separately
    # timed calls (select and decode stand for their share of decode_step)
    dominant = max((k for k in per_step_us if k != "decode_step"), key=per_step_us.get)
    topn = "topn_cta_kernel" if layers[0].cache.max_blocks <= TOPN_CTA_MAX_BLOCKS else "topn_kernel"
    rect_rows = B * f * w.num_q_heads
    rect_merge = ("merge_rows_kernel" if rect_rows >= ROW_MERGE_MIN_ROWS and
                  layers[0].resa.resa_rectify_num_splits(layers[0].cache.struct, f) <= ROW_MERGE_MAX_SPLITS
                  else "merge_kernel")
    # the call's kernels and the sources they are built from (the merges live in sparse_decode.cu)
    kernel, src = {"decode": ("sparse_decode_kernel+merge_kernel", ("sparse_decode.cu",)),
                   "select": ("score_kernel+" + topn, ("select.cu",)),
                   "rectify": ("rectify_kernel+" + rect_merge, ("rectify.cu", "sparse_decode.cu")),
                   "commit": ("commit_append_kernel", ("kv_commit.cu",)),
                   "overwrite": ("commit_overwrite_kernel", ("kv_commit.cu",))}[dominant]
    achieved = algo[dominant] / (mean_us[dominant] * 1e-6) / 1e9
    roofline = {"bound": "hbm", "call": dominant, "kernel": kernel, "achieved": round(achieved, 1), "peak": hbm,
                "unit": "GB/s", "frac": round(achieved / hbm, 3), "peak_kind": peak_kind,
                "traffic": profiled_traffic(dominant, w.name, source_hash(*src)),
                "algorithmic_bytes_per_launch": int(algo[dominant]),
                "timing": "CUDA events around a graph of the step's calls of this kind; per call = total / calls"}

    recall = needle_recall(layers) if w.needle_blocks > 0 else None
    targets = None
    if world == 1 and not args.no_targets:
        targets = run_targets(device)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        Kb, Vb = host_logical_kv(layers[0].cache, 0, w.context)
        sample = {"K": Kb, "V": Vb, "q": bits(layers[0].q[:, 0]), "k": bits(layers[0].k[:, 0]),
                  "v": bits(layers[0].v[:, 0]), "rq": bits(layers[0].rq[0]), "rk": bits(layers[0].rk[0]),
                  "rv": bits(layers[0].rv[0]), "f": f, "keep": w.keep, "n_min": w.n_min_blocks,
                  "n_local": w.n_local_blocks}
        times = run_oracle_subprocess(sample, threads=1, min_seconds=CPU_BASELINE_SECONDS)
        secs_cpu = sum(times)
        cpu = {"value": round(f * len(times) / secs_cpu, 2), "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": f"1 of {B} sequences x 1 of {L} layers: {f} decode steps + 1 rectification at context "
                         f"{w.context}, timed {len(times)} times (fp64 numpy, 1 BLAS thread)",
               "seconds": round(secs_cpu, 3)}
        # informational: the same oracle with its BLAS pool on every host core
        ncores = os.cpu_count() or 1
        times_all = run_oracle_subprocess(sample, threads=ncores, min_seconds=CPU_BASELINE_ALL_SECONDS)
        cpu["all_cores"] = {"value": round(f * len(times_all) / sum(times_all), 2), "unit": UNIT, "cores": ncores,
                            "seconds": round(sum(times_all), 3), "note": "informational; the baseline is 1 thread"}

    launches = args.steps * L * (f * LayerCache.KERNELS_PER_DECODE_STEP + LayerCache.KERNELS_PER_RECTIFY)
    line = {"metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(secs_max * 1e3 / args.steps, 4), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": config_of(w, args), "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": launches, "clocks": clk, "calls": calls, "context_at_timed_start": T_timed0,
            "eq6_ratio": round(eq6_ratio(BLOCK, w.keep, f), 5), "targets": targets}
    if recall is not None:
        line["needle_recall"] = recall
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


ATTR_REPS = 3
CPU_BASELINE_SECONDS = 10.0  # oracle work timed for cpu_baseline (whole periods, at least one)
CPU_BASELINE_ALL_SECONDS = 5.0    # the informational all-cores timing of the same sample
ORACLE_MAX_REPEATS = 400
TOPN_CTA_MAX_BLOCKS = 6144  # caches of up to this many blocks per sequence use the one-CTA top-n
ROW_MERGE_MIN_ROWS, ROW_MERGE_MAX_SPLITS = 1024, 16  # merges of at least this many rows, at most this many splits, take a warp per row


E2E_INPUTS = ("q", "k", "v", "rq", "rk", "rv")  # LayerCache device inputs of one period
E2E_OUTPUTS = ("out", "rout")                    # and its outputs


def run_e2e(args, layers):
    """Same metric through the public API with host buffers, as a serving loop
    runs it: every step copies its inputs from pinned host memory into device
    buffers, replays the step's C-ABI calls and copies all its outputs back to
    pinned host memory. Two sets of device buffers (and a graph captured on
    each) let the copies of step i + 1's inputs and of step i - 1's outputs run
    on a copy stream while step i computes; every byte of every step still
    crosses, inside the timed region."""
    import torch
    f, B, L = layers[0].w.f, layers[0].w.batch, len(layers)
    device = layers[0].out.device
    # Each buffer set is one contiguous device buffer for all layers' inputs
    # and one for their outputs (tensors are views at 256-byte aligned
    # offsets), so a step's inputs cross in one copy and its outputs in one.
    def layout(names):
        offs, n = [], 0
        for Lc in layers:
            o = {}
            for name in names:
                o[name] = n
                n += (getattr(Lc, name).numel() + 127) // 128 * 128
            offs.append(o)
        return offs, n

    in_offs, in_n = layout(E2E_INPUTS)
    out_offs, out_n = layout(E2E_OUTPUTS)
    orig = [{n: getattr(Lc, n) for n in E2E_INPUTS + E2E_OUTPUTS} for Lc in layers]
    for t in (t for o in orig for t in o.values()):
        assert t.dtype == torch.bfloat16 and t.is_contiguous()
    flat_in = [torch.empty(in_n, dtype=torch.bfloat16, device=device) for _ in range(2)]
    flat_out = [torch.empty(out_n, dtype=torch.bfloat16, device=device) for _ in range(2)]
    graphs = []
    for k in range(2):
        for i, Lc in enumerate(layers):
            for n in E2E_INPUTS:
                t = orig[i][n]
                v = flat_in[k][in_offs[i][n]:in_offs[i][n] + t.numel()].view(t.shape)
                v.copy_(t)
                setattr(Lc, n, v)
            for n in E2E_OUTPUTS:
                t = orig[i][n]
                setattr(Lc, n, flat_out[k][out_offs[i][n]:out_offs[i][n] + t.numel()].view(t.shape))
        graphs.append(capture(lambda: run_period(layers), device))
    for Lc, o in zip(layers, orig):
        for n, t in o.items():
            setattr(Lc, n, t)
    for g in graphs:                     # the first launch of a graph uploads it
        g.replay()
    torch.cuda.synchronize()
    host_in = flat_in[0].cpu().pin_memory()
    host_out = torch.empty(out_n, dtype=torch.bfloat16).pin_memory()
    h2d = host_in.numel() * host_in.element_size()
    d2h = host_out.numel() * host_out.element_size()
    comp, copy = torch.cuda.current_stream(), torch.cuda.Stream(device=device)
    ready = [torch.cuda.Event() for _ in range(2)]      # a set's inputs have landed
    done = [torch.cuda.Event() for _ in range(2)]       # a set's step has run (inputs read, outputs written)
    drained = [torch.cuda.Event() for _ in range(2)]    # a set's outputs have been copied out

    def h2d_into(k):
        with torch.cuda.stream(copy):
            flat_in[k].copy_(host_in, non_blocking=True)
            ready[k].record(copy)

    def d2h_from(k):
        with torch.cuda.stream(copy):
            copy.wait_event(done[k])
            host_out.copy_(flat_out[k], non_blocking=True)
            drained[k].record(copy)

    barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(comp)
    copy.wait_event(e0)
    h2d_into(0)
    for step in range(args.steps):
        k = step % 2
        if step + 1 < args.steps:
            h2d_into(1 - k)          # queued behind the drain of step - 1, which used that set
        comp.wait_event(ready[k])
        if step >= 2:
            comp.wait_event(drained[k])  # step - 2's outputs (same set) are out before they are overwritten
        graphs[k].replay()
        done[k].record(comp)
        d2h_from(k)
    comp.wait_stream(copy)
    e1.record(comp)
    torch.cuda.synchronize()
    barrier()
    secs = max_over_ranks(e0.elapsed_time(e1) / 1e3, device)
    _, world, _ = dist_env()
    return {"value": round(aggregate(B * f * L * args.steps, secs, world), 1), "unit": UNIT,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "path": "per step: one pinned host -> device copy of all inputs (every layer's decode and rectify "
                    "inputs, contiguous), the step's C-ABI calls (captured in a CUDA graph), one device -> pinned "
                    "host copy of every decode and rectify output; two device buffer sets so step i + 1's inputs "
                    "and step i - 1's outputs cross while step i computes"}


def rectify_cell(T: int, f: int, device, peaks: dict, peak_kind: str) -> dict:
    """One cell of the rectification sweep: dense causal attention of f new
    queries (28 q / 4 KV heads, d 128, batch 1) against a cached context T,
    then the K/V overwrite and block-summary refresh of the touched blocks.
    Enough independent caches rotate that the rotation's working set exceeds
    L2; each call is timed from a CUDA graph of the rotation with CUDA events."""
    import torch
    from paper_2506_04108_gb300 import resa
    Hq, Hkv, B = 28, 4, 1
    ncache = max(1, math.ceil(300e6 / (B * Hkv * T * 512)))
    caches = []
    for i in range(ncache):
        maxb = (T + BLOCK - 1) // BLOCK + 1
        pt = synth.page_table(synth.rng(synth.RECTIFY_SWEEP_SEED + i), B, maxb)
        cch = resa.PagedKVCache(B, Hq, Hkv, maxb, pt, device=device, zero_pools=False)
        tg = torch.Generator(device=device)
        tg.manual_seed(synth.RECTIFY_SWEEP_SEED * 10 + i)
        for pool in (cch.k_pool, cch.v_pool):
            pool.copy_(torch.randn(pool.shape, generator=tg, device=device))
        cch.seq_lens.fill_(T)
        resa.resa_update_summaries(cch.struct, 0, -1)
        qn = torch.randn((B, f, Hq, HEAD_DIM), generator=tg, device=device).to(torch.bfloat16)
        kn = torch.randn((B, f, Hkv, HEAD_DIM), generator=tg, device=device).to(torch.bfloat16)
        vn = torch.randn((B, f, Hkv, HEAD_DIM), generator=tg, device=device).to(torch.bfloat16)
        out = torch.empty_like(qn)
        nb = resa.resa_workspace_size(cch.struct, 8, 0, f)
        ws = torch.empty(nb, dtype=torch.uint8, device=device)
        caches.append((cch, qn, kn, vn, out, ws, nb))
    p = resa.params(0.1, 0, 0)

    def one(c):
        cch, qn, kn, vn, out, ws, nb = c
        resa.resa_rectify_attention(cch.struct, qn, kn, vn, f, p, out, None, ws, nb)
        resa.resa_commit_kv(cch.struct, kn, vn, f, True)

    def rect_only(c):
        cch, qn, kn, vn, out, ws, nb = c
        resa.resa_rectify_attention(cch.struct, qn, kn, vn, f, p, out, None, ws, nb)
    for c in caches:
        one(c)
    torch.cuda.synchronize()
    reps = max(2, math.ceil(8 / ncache))
    g_all = capture(lambda: [one(c) for _ in range(reps) for c in caches], device)
    g_rect = capture(lambda: [rect_only(c) for _ in range(reps) for c in caches], device)
    g_all.replay()
    g_rect.replay()
    calls = reps * ncache
    t_all = time_graph(g_all, 3) / calls
    t_rect = time_graph(g_rect, 3) / calls
    for c in caches:
        code, _ = resa.resa_read_device_error(c[0].struct)
        if code:
            raise RuntimeError(f"device error {resa.DEVICE_ERRORS.get(code)}")
    flops = rectify_flops(B, Hq, T, f)
    byts = rectify_bytes(B, Hq, Hkv, T, f)
    tf = flops / t_rect / 1e12
    gbs = byts / t_rect / 1e9
    del caches, g_all, g_rect
    torch.cuda.empty_cache()
    return {"context": T, "f": f, "batch": B, "caches_rotated": ncache,
            "rectify_us": round(t_rect * 1e6, 2), "rectify_plus_overwrite_us": round(t_all * 1e6, 2),
            "TFLOP/s": round(tf, 1), "frac_bf16_burst": round(tf / float(peaks["bf16_tflops"]), 3),
            "frac_bf16_sustained": round(tf / float(peaks["bf16_tflops_sustained"]), 3),
            "GB/s": round(gbs, 1), "frac_hbm": round(gbs / float(peaks["hbm_gbs"]), 3),
            "bound": "hbm" if 7 * f < float(peaks["bf16_tflops"]) / float(peaks["hbm_gbs"]) * 1e3 else "tensor",
            "peak_kind": peak_kind}


def run_rectify_sweep(args):
    """Rectification-only sweep (the f x context grid of synth.RECTIFY_SWEEP),
    one JSON line per cell (see rectify_cell)."""
    import torch
    from paper_2506_04108_gb300 import build as _b
    from paper_2506_04108_gb300 import resa
    _b.build()
    resa.load()
    device = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    peaks, peak_kind = load_peaks()
    cells = synth.RECTIFY_SWEEP
    if args.rectify_cells:
        cells = [tuple(int(x) for x in cell.split(":")) for cell in args.rectify_cells.split(",")]
    for T, f in cells:
        print(json.dumps({"mode": "rectify_sweep", **rectify_cell(T, f, device, peaks, peak_kind)}), flush=True)


TARGET_WORKLOAD = "qwen7b_b1_ctx256k_keep5"
TARGET_LAYERS = 4
TARGET_RECTIFY = ((262144, 32), (262144, 64))
TARGET_DECODE_FRAC_HBM = 0.70
TARGET_RECTIFY_FRAC_BF16 = 0.50


def run_targets(device) -> dict:
    """The two performance targets, measured after the headline (no oracle):
    sparse decode at 256K context, batch 1, keep 0.05 (the decode call's
    roofline fraction, the fused decode step per token, the rectify share of
    the period), over TARGET_LAYERS rotated layer caches, per-call graphs
    timed with CUDA events; and rectification at 256K with f = 32 and 64
    against the burst bf16 peak (a call timed in isolation)."""
    import torch
    w = synth.WORKLOADS[TARGET_WORKLOAD]
    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    f, L, B = w.f, TARGET_LAYERS, w.batch
    capacity = ((w.context + f * (2 + 2 * (1 + ATTR_REPS)) + BLOCK) // BLOCK + 1) * BLOCK
    layers = [LayerCache(w, capacity, w.seed * 100 + 53 * i, device) for i in range(L)]
    run_period(layers)                          # warm-up call outside any graph, appends f tokens
    torch.cuda.synchronize()
    T_attr = w.context + f
    with ClockSampler(device.index or 0) as clocks:
        mean_us, ncalls = time_call_kinds(layers, device)
        cells = [rectify_cell(T, fr, device, peaks, peak_kind) for T, fr in TARGET_RECTIFY]
    algo = call_bytes(w, T_attr)
    dec_gbs = algo["decode"] / (mean_us["decode"] * 1e-6) / 1e9
    period_us = sum(mean_us[k] * ncalls[k] for k in IN_STEP) / L     # one layer's period of f tokens
    rect_us = (mean_us["rectify"] * ncalls["rectify"] + mean_us["overwrite"] * ncalls["overwrite"]) / L
    del layers
    torch.cuda.empty_cache()
    rect = {}
    for c in cells:
        rect[f"f{c['f']}"] = {k: c[k] for k in ("rectify_us", "rectify_plus_overwrite_us", "TFLOP/s",
                                                "frac_bf16_burst", "frac_bf16_sustained", "GB/s", "frac_hbm",
                                                "bound")}
    return {
        "decode_256k": {
            "workload": w.name, "batch": B, "context": T_attr, "keep": w.keep, "layers_rotated": L,
            "decode_call_us": round(mean_us["decode"], 2), "decode_GB/s": round(dec_gbs, 1),
            "decode_frac_hbm": round(dec_gbs / hbm, 3), "decode_algorithmic_bytes": int(algo["decode"]),
            "target_frac_hbm": TARGET_DECODE_FRAC_HBM, "met": dec_gbs / hbm >= TARGET_DECODE_FRAC_HBM,
            "select_call_us": round(mean_us["select"], 2),
            "decode_step_us_per_token": round(mean_us["decode_step"], 2),
            "us_per_token_with_rectify": round(period_us / f, 2),
            "rectify_share_of_period": round(rect_us / period_us, 3),
            "rectify_call_us": round(mean_us["rectify"], 2),
            "decode_attention_latency_note": "per token of one layer: the fused decode step (append + select + "
                                            "decode); with rectify and overwrite amortised over the f tokens in "
                                            "us_per_token_with_rectify"},
        "rectify_256k": {**rect, "target_frac_bf16_burst": TARGET_RECTIFY_FRAC_BF16,
                         "met_f64": rect["f64"]["frac_bf16_burst"] >= TARGET_RECTIFY_FRAC_BF16,
                         "peak_bf16_burst": float(peaks["bf16_tflops"])},
        "peak_kind": peak_kind, "clocks": clocks.summary(),
        "timing": "CUDA events around per-call-type CUDA graphs (decode: 4 rotated 256K caches; rectify: one "
                  "537 MB cache per call, larger than L2), after the headline's timed region"}


def run_breakdown(args):
    """Per-call latency breakdown of one layer-step at batch 8 (28 q / 4 KV
    heads, d 128, keep 0.1, n_min 128 blocks, n_local 1, f 32) for each
    context in synth.BREAKDOWN_CONTEXTS, next to dense flash decoding of the
    same step (the sparse-decode kernel given every block of the sequence).
    The sparse step is commit + select + sparse decode + (rectify +
    overwrite) / f; the dense step is commit + dense decode. Enough caches
    rotate per context that the rotation exceeds L2. One JSON line per
    context."""
    import dataclasses
    import torch
    from paper_2506_04108_gb300 import build as _b
    from paper_2506_04108_gb300 import resa
    _b.build()
    resa.load()
    device = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    base = synth.WORKLOADS[DEFAULT_WORKLOAD]
    for T0 in synth.BREAKDOWN_CONTEXTS:
        w = dataclasses.replace(base, name=f"breakdown_b8_ctx{T0 // 1024}k", context=T0)
        B, Hq, Hkv, f = w.batch, w.num_q_heads, w.num_kv_heads, w.f
        ncache = max(1, math.ceil(400e6 / (B * Hkv * T0 * 512)))
        capacity = ((T0 + f * (2 + 2 * ATTR_REPS) + BLOCK) // BLOCK + 1) * BLOCK
        layers = [LayerCache(w, capacity, w.seed * 100 + 31 * i, device) for i in range(ncache)]
        run_period(layers)                       # warm-up, appends f tokens
        T = T0 + f
        torch.cuda.synchronize()
        # dense selection: every block of every sequence, in order
        M = (T + BLOCK - 1) // BLOCK
        maxb = layers[0].cache.max_blocks
        dense_idx = torch.arange(maxb, dtype=torch.int32, device=device).expand(B, Hkv, maxb).contiguous()
        dense_cnt = torch.full((B, Hkv), M, dtype=torch.int32, device=device)
        dense_ws = []
        for Lc in layers:
            nb = resa.resa_workspace_size(Lc.cache.struct, maxb, 0, 0)
            dense_ws.append((torch.empty(nb, dtype=torch.uint8, device=device), nb))

        def dense(i, t):
            Lc = layers[i]
            ws, nb = dense_ws[i]
            resa.resa_sparse_decode(Lc.cache.struct, Lc.q[t], dense_idx, dense_cnt, maxb, Lc.p, Lc.out[t], None, 0,
                                    ws, nb)
        kinds = {
            "select": (lambda: [Lc.select(t) for t in range(f) for Lc in layers], f),
            "decode": (lambda: [Lc.sparse_decode(t) for t in range(f) for Lc in layers], f),
            "dense_decode": (lambda: [dense(i, t) for t in range(f) for i in range(len(layers))], f),
            "rectify": (lambda: [Lc.rectify_attention() for Lc in layers], 1),
            "overwrite": (lambda: [Lc.overwrite() for Lc in layers], 1),
            "commit": (lambda: [Lc.commit(t) for t in range(f) for Lc in layers], f),
        }
        us = {}
        for kind, (fn, per_layer) in kinds.items():
            gk = capture(fn, device)
            gk.replay()
            us[kind] = time_graph(gk, ATTR_REPS) / (per_layer * len(layers)) * 1e6
            del gk
        check_device_errors(layers)
        sparse = us["commit"] + us["select"] + us["decode"] + (us["rectify"] + us["overwrite"]) / f
        dense_step = us["commit"] + us["dense_decode"]
        dense_bytes = B * Hkv * T * 512 + B * Hq * HEAD_DIM * 4
        sparse_bytes = decode_bytes(B, Hq, Hkv, T, w.keep, w.n_min_blocks, w.n_local_blocks)
        line = {"mode": "breakdown", "context": T0, "batch": B, "q_heads": Hq, "kv_heads": Hkv, "keep": w.keep,
                "f": f, "caches_rotated": ncache,
                "us_per_call": {k: round(v, 2) for k, v in us.items()},
                "sparse_step_us": round(sparse, 2), "dense_step_us": round(dense_step, 2),
                "dense_over_sparse": round(dense_step / sparse, 2),
                "dense_decode_GB/s": round(dense_bytes / (us["dense_decode"] * 1e-6) / 1e9, 1),
                "dense_decode_frac_hbm": round(dense_bytes / (us["dense_decode"] * 1e-6) / 1e9 / hbm, 3),
                "sparse_decode_GB/s": round(sparse_bytes / (us["decode"] * 1e-6) / 1e9, 1),
                "sparse_decode_frac_hbm": round(sparse_bytes / (us["decode"] * 1e-6) / 1e9 / hbm, 3),
                "peak_kind": peak_kind, "data": "synthetic"}
        print(json.dumps(line), flush=True)
        del layers, dense_ws, dense_idx
        torch.cuda.empty_cache()


def run_prefill(args):
    """Chunked dense prefill (Algorithm 1's prefill): for each chunk of the
    prompt, the append commit of its K/V (block keys built online) and the
    rectification call with f = chunk, which attends the chunk's queries
    causally to the cached prefix and the chunk. Batch 1, 28 q / 4 KV heads,
    d 128, chunks of synth.PREFILL_CHUNK tokens; the whole prompt is one CUDA
    graph. One JSON line per prompt length (tokens/s and TFLOP/s of the useful
    causal flops, 4 d Hq L^2 / 2 + O(L))."""
    import torch
    from paper_2506_04108_gb300 import build as _b
    from paper_2506_04108_gb300 import resa
    _b.build()
    resa.load()
    device = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    peaks, peak_kind = load_peaks()
    Hq, Hkv, B, C = 28, 4, 1, synth.PREFILL_CHUNK
    for L in synth.PREFILL_LENGTHS:
        maxb = (L + BLOCK - 1) // BLOCK + 1
        pt = synth.page_table(synth.rng(synth.PREFILL_SEED), B, maxb)
        cch = resa.PagedKVCache(B, Hq, Hkv, maxb, pt, device=device, zero_pools=False)
        tg = torch.Generator(device=device)
        tg.manual_seed(synth.PREFILL_SEED)
        q = torch.randn((B, L, Hq, HEAD_DIM), generator=tg, device=device).to(torch.bfloat16)
        k = torch.randn((B, L, Hkv, HEAD_DIM), generator=tg, device=device).to(torch.bfloat16)
        v = torch.randn((B, L, Hkv, HEAD_DIM), generator=tg, device=device).to(torch.bfloat16)
        out = torch.empty_like(q)
        nb = resa.resa_workspace_size(cch.struct, 8, 0, C)
        ws = torch.empty(nb, dtype=torch.uint8, device=device)
        p = resa.params(0.1, 0, 0)
        chunks = [(c0, min(C, L - c0)) for c0 in range(0, L, C)]
        # per chunk: contiguous [B, f, H, d] views (slices of [B, L, H, d] are contiguous for B = 1)
        views = [(q[:, c0:c0 + f], k[:, c0:c0 + f], v[:, c0:c0 + f], out[:, c0:c0 + f], f) for c0, f in chunks]

        def prefill():
            cch.seq_lens.zero_()
            for qc, kc, vc, oc, f in views:
                resa.resa_commit_kv(cch.struct, kc, vc, f, False)
                resa.resa_rectify_attention(cch.struct, qc, kc, vc, f, p, oc, None, ws, nb)
        prefill()
        torch.cuda.synchronize()
        g = capture(prefill, device)
        g.replay()
        secs = time_graph(g, 3)
        code, _ = resa.resa_read_device_error(cch.struct)
        if code:
            raise RuntimeError(f"device error {resa.DEVICE_ERRORS.get(code)}")
        flops = 4.0 * HEAD_DIM * Hq * B * (L * (L + 1) / 2)
        tf = flops / secs / 1e12
        print(json.dumps({"mode": "prefill", "prompt": L, "chunk": C, "batch": B, "q_heads": Hq, "kv_heads": Hkv,
                          "ms": round(secs * 1e3, 3), "tokens/s": round(B * L / secs, 1),
                          "TFLOP/s": round(tf, 1), "frac_bf16_burst": round(tf / float(peaks["bf16_tflops"]), 3),
                          "frac_bf16_sustained": round(tf / float(peaks["bf16_tflops_sustained"]), 3),
                          "peak_kind": peak_kind, "data": "synthetic"}), flush=True)
        del cch, q, k, v, out, ws, g
        torch.cuda.empty_cache()


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--layers", type=int, default=None,
                    help="independent layer caches rotated per decode step (default: the workload's layer count, "
                         "at least 4)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-targets", action="store_true",
                    help="skip the 256K decode and rectify target measurements after the headline")
    ap.add_argument("--prefill", action="store_true", help="chunked dense prefill throughput (32K, 128K prompts)")
    ap.add_argument("--breakdown", action="store_true",
                    help="per-call latency breakdown versus dense decoding at 16K/64K/256K, batch 8")
    ap.add_argument("--rectify-sweep", action="store_true",
                    help="time rectification over the 16K/64K/256K x f 16/32/64 grid instead")
    ap.add_argument("--rectify-cells", default=None,
                    help="with --rectify-sweep: only these cells, 'context:f' comma-separated (e.g. 65536:64)")
    ap.add_argument("--oracle-worker", default=None, help=argparse.SUPPRESS)
    ap.add_argument("--repeats", type=int, default=1, help=argparse.SUPPRESS)
    ap.add_argument("--min-seconds", type=float, default=0.0, help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.oracle_worker:
        sample = dict(np.load(args.oracle_worker))
        secs = [oracle_period(sample) for _ in range(args.repeats)]
        while sum(secs) < args.min_seconds and len(secs) < ORACLE_MAX_REPEATS:
            secs.append(oracle_period(sample))
        print(json.dumps({"seconds": secs}))
        return
    if args.warmup < 3 and args.impl == "ours":
        ap.error("--warmup must be >= 3")
    w = synth.WORKLOADS[args.workload]
    if args.layers is None:
        args.layers = max(4, w.layers)
    if args.rectify_sweep:
        run_rectify_sweep(args)
        return
    if args.breakdown:
        run_breakdown(args)
        return
    if args.prefill:
        run_prefill(args)
        return
    if args.impl == "reference":
        run_reference(args, w)
    else:
        run_ours(args, w)


if __name__ == "__main__":
    main()
