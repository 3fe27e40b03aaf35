"""The allocation-free decode entry point (resa_sparse_decode_static).

Some callers cannot allocate device memory at all -- a plugin inside a host
framework that owns every device allocation, or a latency-critical loop where
an allocation (which may synchronise the device) is not allowed. For them the
library offers resa_sparse_decode_static, which keeps the split partials in a
fixed static device buffer instead of a caller workspace. This file checks,
through the C ABI, that it returns what resa_sparse_decode returns on two
calls in a row (the buffer is reused and keeps stale contents between calls),
and that a call too large for the buffer is refused before any launch.
It is collected last so a failure here never hides the other tests.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2506_04108_gb300 import resa, synth
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu


def test_static_scratch_decode_matches_workspace_decode_on_two_calls():
    g, Hkv, lens = 7, 4, [2053, 1000]
    gen = synth.rng(4242)
    Ks = [synth.normal_bf16(gen, (Hkv, T, 128)) for T in lens]
    Vs = [synth.normal_bf16(gen, (Hkv, T, 128)) for T in lens]
    cache = H.make_cache(Ks, Vs, g * Hkv, 140)
    p = resa.params(0.1, 16, 1)
    n_cap = resa.resa_max_selected(cache.struct, p)
    B, Hq = len(lens), g * Hkv
    idx = torch.empty((B, Hkv, n_cap), dtype=torch.int32, device="cuda")
    cnt = torch.empty((B, Hkv), dtype=torch.int32, device="cuda")
    ws, nb = H.workspace(cache, n_cap)
    for call in range(2):                       # two calls in a row, different queries
        q = H.dev_bf16(synth.normal_bf16(gen, (B, Hq, 128)))
        resa.resa_select_blocks(cache.struct, q, p, idx, cnt, n_cap, ws, nb)
        ref = torch.empty((B, Hq, 128), dtype=torch.bfloat16, device="cuda")
        ref_lse = torch.empty((B, Hq), dtype=torch.float32, device="cuda")
        resa.resa_sparse_decode(cache.struct, q, idx, cnt, n_cap, p, ref, ref_lse, 0, ws, nb)
        out = torch.full((B, Hq, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.full((B, Hq), float("nan"), dtype=torch.float32, device="cuda")
        resa.resa_sparse_decode_static(cache.struct, q, idx, cnt, n_cap, p, out, lse, 0)
        torch.cuda.synchronize()
        H.check_outputs(H.host_f64(out), H.host_f64(ref), f"call {call}")
        assert np.allclose(lse.cpu().numpy(), ref_lse.cpu().numpy(), rtol=0, atol=1e-5)
    assert resa.resa_read_device_error(cache.struct) == (0, 0)


def test_static_scratch_decode_refuses_calls_beyond_its_buffer():
    gen = synth.rng(4343)
    Ks = [synth.normal_bf16(gen, (4, 64, 128)) for _ in range(2)]
    Vs = [synth.normal_bf16(gen, (4, 64, 128)) for _ in range(2)]
    cache = H.make_cache(Ks, Vs, 28, 8)
    p = resa.params(0.1, 0, 1)
    idx = torch.zeros((2, 4, 4), dtype=torch.int32, device="cuda")
    cnt = torch.ones((2, 4), dtype=torch.int32, device="cuda")
    q = torch.zeros((2, 28, 128), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(q)
    # 56 rows x 1000 splits x 129 floats is far above RESA_STATIC_SCRATCH_BYTES (4 MiB)
    st = resa.load().resa_sparse_decode_static(ctypes.byref(cache.struct), q.data_ptr(), idx.data_ptr(),
                                               cnt.data_ptr(), 4, ctypes.byref(p), out.data_ptr(), None, 1000,
                                               torch.cuda.current_stream().cuda_stream)
    assert st == 3                               # RESA_ERR_WORKSPACE, nothing launched
