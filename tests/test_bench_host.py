"""Host-side logic of bench.py (CPU only): the algorithmic byte model against
Eq. 6, the multi-rank aggregation over a world_size-2 gloo group, and the
timing loop of the CPU baseline."""
import json
import math
import os

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2506_04108_gb300 import synth


def test_step_bytes_follow_eq6():
    """Per decode step: summaries (1/b of the KV cache) + selected KV (keep) +
    amortised rectification (1/f) ~= Eq. 6 times the KV bytes. The small
    extra terms (fp32 scores, queries, outputs, partial last block) stay
    within 3%."""
    B, Hq, Hkv, T, f = 8, 28, 4, 32768, 32
    kv = B * Hkv * T * 2 * 128 * 2
    M = T // 16
    per_step = (bench.select_bytes(B, Hq, Hkv, T, 0.1, 0, 1) + bench.decode_bytes(B, Hq, Hkv, T, 0.1, 0, 1)
                + bench.rectify_bytes(B, Hq, Hkv, T, f) / f)
    ratio = per_step / kv
    assert math.isclose(bench.eq6_ratio(16, 0.1, 32), 0.19375)
    assert abs(ratio - bench.eq6_ratio(16, 0.1, 32)) / 0.19375 < 0.03
    assert bench.budget(M, 0.1, 128, 1) == 205


def test_decode_bytes_count_valid_tokens_of_partial_block():
    # T = 33: M = 3 blocks, all kept; 33 tokens attended
    assert bench.decode_bytes(1, 1, 1, 33, 1.0, 0, 1) == 33 * 512 + 2 * 256


def test_rectify_flops_causal_count():
    # f = 2 rows at T = 10: row 0 sees 9 keys, row 1 sees 10
    assert bench.rectify_flops(1, 1, 10, 2) == 4 * 128 * (9 + 10)


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    r, w = bench.init_dist("gloo")
    bench.barrier()
    secs = 1.0 + rank                      # rank 1 is the slow one
    m = bench.max_over_ranks(secs)
    q.put((r, w, m, bench.aggregate(100.0, m, w)))
    dist.destroy_process_group()


def test_two_rank_gloo_aggregation():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = 29500 + (os.getpid() % 1000)
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r, (rank, world, m, value) in enumerate(res):
        assert rank == r and world == 2
        assert m == pytest.approx(2.0)          # max over ranks
        assert value == pytest.approx(100.0 * 2 / 2.0)


def test_single_process_helpers_are_identity():
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.aggregate(10.0, 2.0, 1) == 5.0


def test_oracle_worker_times_whole_periods_until_min_seconds():
    """cpu_baseline's timing loop: at least the requested periods, then more
    until the timed work reaches min_seconds (a small 4K-shaped sample)."""
    w = synth.WORKLOADS["b1_h8kv2_ctx4k_f8"]
    s = bench.host_sample(w, 512)
    times = bench.run_oracle_subprocess(s, threads=1, repeats=2, min_seconds=0.5)
    assert len(times) >= 2 and all(t > 0 for t in times)
    assert sum(times) >= 0.5 or len(times) == bench.ORACLE_MAX_REPEATS
    assert sum(times[:-1]) < 0.5 or len(times) == 2  # stops at the first period past the bound


def test_clock_summary_keeps_the_timed_window(tmp_path):
    """The clock summary uses only the samples inside begin()/end() when any
    fell there (an idle sample before the region and a throttled one after it
    are left out), and all of them otherwise."""
    import datetime as dt
    t0 = dt.datetime(2026, 1, 2, 3, 4, 5)
    rows = [(t0, 1200, ""), (t0 + dt.timedelta(seconds=1), 2070, ""), (t0 + dt.timedelta(seconds=1.02), 2070, ""),
            (t0 + dt.timedelta(seconds=3), 1500, "Active")]

    def sampler(window):
        path = tmp_path / f"clk{window is not None}.csv"
        with open(path, "w") as fh:
            for t, mhz, slow in rows:
                fh.write(f"{t:%Y/%m/%d %H:%M:%S.%f}, 0, {mhz}, 2070, 900.0, 0x0, "
                         f"{slow or 'Not Active'}, Not Active, Not Active, Not Active\n")
        c = bench.ClockSampler(0)
        c.proc, c.path, c.window = object(), str(path), window
        return c.summary()

    inside = sampler([t0 + dt.timedelta(seconds=0.5), t0 + dt.timedelta(seconds=2)])
    assert inside == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 2, "window": "timed region"}
    everything = sampler(None)
    assert everything["samples"] == 4 and everything["window"] == "all samples"
    assert everything["reasons"] == ["hw_slowdown"] and everything["sm_mhz"] == 1785.0


def test_profiled_traffic_needs_the_current_source_hash(tmp_path, monkeypatch):
    """The roofline's `traffic` comes from a committed ncu summary only while
    the kernel sources it was taken from are unchanged (a stale entry gives
    None); a call built from two sources hashes both."""
    h_dec = bench.source_hash("sparse_decode.cu")
    h_rect = bench.source_hash("rectify.cu", "sparse_decode.cu")
    assert h_rect != bench.source_hash("rectify.cu")
    table = {"decode": {"w": {"dram_bytes_per_call": 123, "source_hash": h_dec}},
             "rectify": {"w": {"dram_bytes_per_call": 456, "source_hash": bench.source_hash("rectify.cu")}}}
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(table))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic("decode", "w", h_dec) == 123
    assert bench.profiled_traffic("rectify", "w", h_rect) is None  # taken before the merge source was hashed too
    assert bench.profiled_traffic("select", "w", h_dec) is None
    assert bench.profiled_traffic("decode", "other workload", h_dec) is None
