"""C-ABI boundary checks that need no GPU: the library builds, loads, exports
every function include/resa.h declares, and rejects invalid arguments on the
host before any CUDA call."""
import ctypes
import os
import re

import pytest

import oracle as O
from paper_2506_04108_gb300 import build, resa

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return resa.load()


def declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        text = open(os.path.join(ROOT, "include", fn)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names |= set(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(resa_\w+)\s*\(", text, flags=re.M))
    return sorted(names)


def test_header_declares_the_five_path_calls():
    names = declared_functions()
    for n in ["resa_update_summaries", "resa_select_blocks", "resa_sparse_decode", "resa_rectify_attention",
              "resa_commit_kv"]:
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 11
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(resa.EXPORTED) == names


def test_abi_version_and_status_strings(lib):
    assert resa.resa_abi_version() == 1
    for code, name in resa.STATUS_NAMES.items():
        assert lib.resa_status_string(code).decode() == name


def fake_cache(**over):
    c = dict(batch=2, num_q_heads=28, num_kv_heads=4, head_dim=128, block_size=16, num_pages=64,
             max_blocks_per_seq=32, reserved0=0, k_pool=0x10000, v_pool=0x20000, page_table=0x30000,
             seq_lens=0x40000, summaries=0x50000, device_status=0x60000)
    c.update(over)
    return resa.ResaCacheT(**c)


P = resa.params(0.1, 16, 1)


@pytest.mark.parametrize("over,code", [
    (dict(batch=0), 1), (dict(num_kv_heads=0), 1), (dict(head_dim=64), 2), (dict(block_size=32), 2),
    (dict(num_q_heads=27), 1), (dict(num_q_heads=64, num_kv_heads=4), 2), (dict(device_status=0), 1),
    (dict(k_pool=0x10008), 1), (dict(page_table=0), 1), (dict(max_blocks_per_seq=0), 1),
])
def test_bad_cache_rejected_on_host(lib, over, code):
    c = fake_cache(**over)
    assert lib.resa_commit_kv(ctypes.byref(c), 0x70000, 0x80000, 1, 0, None) == code
    assert lib.resa_update_summaries(ctypes.byref(c), 0, -1, None) == code


def test_bad_call_arguments_rejected_on_host(lib):
    c = fake_cache()
    cp = ctypes.byref(c)
    assert lib.resa_commit_kv(cp, 0x70000, 0x80000, -1, 0, None) == 1
    assert lib.resa_commit_kv(cp, 0, 0x80000, 1, 0, None) == 1
    assert lib.resa_commit_kv(cp, 0x70000, 0x80000, 1, 2, None) == 1
    assert lib.resa_commit_kv(cp, 0x70008, 0x80000, 1, 0, None) == 1      # misaligned
    assert lib.resa_update_summaries(cp, -1, -1, None) == 1
    assert lib.resa_update_summaries(cp, 5, 3, None) == 1
    assert lib.resa_update_summaries(cp, 0, 33, None) == 1
    bad_keep = resa.params(1.5, 16, 1)
    assert lib.resa_select_blocks(cp, 0x70000, ctypes.byref(bad_keep), 0x1000, 0x2000, 10, 0x3000, 1 << 20,
                                  None) == 1
    neg = resa.params(0.1, -1, 1)
    assert lib.resa_select_blocks(cp, 0x70000, ctypes.byref(neg), 0x1000, 0x2000, 10, 0x3000, 1 << 20, None) == 1
    assert lib.resa_select_blocks(cp, 0x70000, ctypes.byref(P), 0x1000, 0x2000, 0, 0x3000, 1 << 20, None) == 1
    # workspace too small for the fp32 scores (2 * 4 * 32 floats)
    assert lib.resa_select_blocks(cp, 0x70000, ctypes.byref(P), 0x1000, 0x2000, 10, 0x3000, 16, None) == 3
    assert lib.resa_select_blocks(cp, 0x70000, ctypes.byref(P), 0x1000, 0x2000, 10, 0, 1 << 20, None) == 3
    assert lib.resa_sparse_decode(cp, 0x70000, 0x1000, 0x2000, 0, ctypes.byref(P), 0x4000, None, 0, 0x3000,
                                  1 << 20, None) == 1
    assert lib.resa_sparse_decode(cp, 0x70000, 0x1000, 0x2000, 10, ctypes.byref(P), 0, None, 0, 0x3000, 1 << 20,
                                  None) == 1
    assert lib.resa_rectify_attention(cp, 0x70000, 0x71000, 0x72000, 0, ctypes.byref(P), 0x4000, None, 0x3000,
                                      1 << 20, None) == 1
    assert lib.resa_rectify_attention(cp, 0x70000, 0, 0x72000, 8, ctypes.byref(P), 0x4000, None, 0x3000,
                                      1 << 20, None) == 1
    # fused decode step: argument checks precede any CUDA call (explicit splits)
    def step(k=0x70000, v=0x71000, q=0x72000, n_cap=10, out=0x4000, splits=4, ws=0x3000, wsb=1 << 20):
        return lib.resa_decode_step(cp, k, v, q, ctypes.byref(P), 0x1000, 0x2000, n_cap, out, None, splits, ws, wsb,
                                    None)
    assert step(k=0) == 1 and step(v=0) == 1 and step(q=0) == 1 and step(out=0) == 1
    assert step(v=0x71008) == 1 and step(n_cap=0) == 1 and step(splits=-1) == 1 and step(splits=2000) == 1
    assert step(wsb=16) == 3 and step(ws=0) == 3
    # split query of the rectification: f outside [1, capacity] or no output pointer
    n = ctypes.c_int32(0)
    assert lib.resa_rectify_num_splits(cp, 0, ctypes.byref(n)) == 1
    assert lib.resa_rectify_num_splits(cp, 32 * 16 + 1, ctypes.byref(n)) == 1
    assert lib.resa_rectify_num_splits(cp, 8, None) == 1


def test_decode_wait_limit_setter_needs_no_device(lib):
    assert lib.resa_set_decode_wait_polls(0) == 0
    assert lib.resa_set_decode_wait_polls(resa.DEFAULT_DECODE_WAIT_POLLS) == 0


@pytest.mark.parametrize("max_blocks,keep,n_min,n_local", [(256, 0.1, 16, 4), (2048, 0.1, 128, 1),
                                                           (16384, 0.05, 128, 1), (16401, 0.05, 128, 1),
                                                           (10, 0.1, 16, 1), (300, 0.1, 16, 40), (2560, 0.1, 0, 0)])
def test_max_selected_matches_oracle_budget(lib, max_blocks, keep, n_min, n_local):
    c = fake_cache(max_blocks_per_seq=max_blocks, num_pages=2 * max_blocks)
    assert resa.resa_max_selected(c, resa.params(keep, n_min, n_local)) == \
        O.selection_budget(max_blocks, keep, n_min, n_local)


def test_read_device_error_rejects_null(lib):
    c = fake_cache(device_status=0)
    assert lib.resa_read_device_error(ctypes.byref(c), None, None, None) == 1
