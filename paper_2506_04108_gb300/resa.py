"""Thin ctypes binding of libresa (C ABI in include/resa.h).

Argument marshalling only: every function here converts tensors to device
pointers and the current torch stream to a cudaStream_t, calls the C entry
point of the same name, and raises :class:`ResaError` on a non-OK status.
There is no fallback: if ``libresa.so`` has not been built the first call
raises.

:class:`PagedKVCache` owns the caller-side device buffers of one cache (paged
K/V pools, page table, sequence lengths, block summaries, device status) as
torch tensors and exposes them as a ``resa_cache_t``.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int32, c_size_t, c_void_p

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libresa.so")
_lib = None

RESA_OK = 0
STATUS_NAMES = {0: "RESA_OK", 1: "RESA_ERR_INVALID_ARG", 2: "RESA_ERR_UNSUPPORTED", 3: "RESA_ERR_WORKSPACE",
                4: "RESA_ERR_CUDA", 5: "RESA_ERR_DEVICE"}
DEVICE_ERRORS = {0: "RESA_DEV_OK", 1: "RESA_DEV_SEQ_LEN_RANGE", 2: "RESA_DEV_PAGE_RANGE",
                 3: "RESA_DEV_BUDGET_OVER_CAP", 4: "RESA_DEV_WAIT_TIMEOUT", 5: "RESA_DEV_BAD_INDEX"}
EXPORTED = ["resa_abi_version", "resa_status_string", "resa_max_selected", "resa_decode_num_splits",
            "resa_workspace_size", "resa_update_summaries", "resa_commit_kv", "resa_select_blocks",
            "resa_sparse_decode", "resa_rectify_attention", "resa_read_device_error", "resa_sparse_decode_static",
            "resa_commit_kv_active", "resa_rectify_attention_active", "resa_decode_step",
            "resa_rectify_num_splits", "resa_set_decode_wait_polls"]
DEFAULT_DECODE_WAIT_POLLS = 1 << 22


class ResaError(RuntimeError):
    def __init__(self, status: int, call: str, detail: str = ""):
        self.status = status
        super().__init__(f"{call} -> {STATUS_NAMES.get(status, status)}{(': ' + detail) if detail else ''}")


class ResaCacheT(ctypes.Structure):
    _fields_ = [("batch", c_int32), ("num_q_heads", c_int32), ("num_kv_heads", c_int32), ("head_dim", c_int32),
                ("block_size", c_int32), ("num_pages", c_int32), ("max_blocks_per_seq", c_int32),
                ("reserved0", c_int32), ("k_pool", c_void_p), ("v_pool", c_void_p), ("page_table", c_void_p),
                ("seq_lens", c_void_p), ("summaries", c_void_p), ("device_status", c_void_p)]


class ResaParamsT(ctypes.Structure):
    _fields_ = [("keep_ratio", c_double), ("n_min_blocks", c_int32), ("n_local_blocks", c_int32),
                ("sm_scale", c_float), ("reserved0", c_int32)]


def lib_path() -> str:
    return _LIB_PATH


def load() -> ctypes.CDLL:
    """Load libresa.so (built in-tree); raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"{_LIB_PATH} is not built; run `python -m paper_2506_04108_gb300.build`")
    L = ctypes.CDLL(_LIB_PATH)
    cp, pc, pp = POINTER(ResaCacheT), POINTER(ResaParamsT), c_void_p
    sig = {
        "resa_abi_version": ([], c_int32),
        "resa_status_string": ([c_int32], ctypes.c_char_p),
        "resa_max_selected": ([cp, pc, POINTER(c_int32)], c_int32),
        "resa_decode_num_splits": ([cp, c_int32, POINTER(c_int32)], c_int32),
        "resa_rectify_num_splits": ([cp, c_int32, POINTER(c_int32)], c_int32),
        "resa_set_decode_wait_polls": ([ctypes.c_uint32], c_int32),
        "resa_workspace_size": ([cp, c_int32, c_int32, c_int32, POINTER(c_size_t)], c_int32),
        "resa_update_summaries": ([cp, c_int32, c_int32, pp], c_int32),
        "resa_commit_kv": ([cp, pp, pp, c_int32, c_int32, pp], c_int32),
        "resa_select_blocks": ([cp, pp, pc, pp, pp, c_int32, pp, c_size_t, pp], c_int32),
        "resa_sparse_decode": ([cp, pp, pp, pp, c_int32, pc, pp, pp, c_int32, pp, c_size_t, pp], c_int32),
        "resa_rectify_attention": ([cp, pp, pp, pp, c_int32, pc, pp, pp, pp, c_size_t, pp], c_int32),
        "resa_read_device_error": ([cp, POINTER(c_int32), POINTER(c_int32), pp], c_int32),
        "resa_sparse_decode_static": ([cp, pp, pp, pp, c_int32, pc, pp, pp, c_int32, pp], c_int32),
        "resa_commit_kv_active": ([cp, pp, pp, pp, c_int32, c_int32, pp], c_int32),
        "resa_rectify_attention_active": ([cp, pp, pp, pp, pp, c_int32, pc, pp, pp, pp, c_size_t, pp], c_int32),
        "resa_decode_step": ([cp, pp, pp, pp, pc, pp, pp, c_int32, pp, pp, c_int32, pp, c_size_t, pp], c_int32),
    }
    for name, (args, ret) in sig.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = ret
    _lib = L
    return L


def _ptr(x) -> int | None:
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    return int(x)


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        if torch.cuda.is_available():
            return torch.cuda.current_stream().cuda_stream
        return None
    if hasattr(stream, "cuda_stream"):
        return stream.cuda_stream
    return int(stream)


def _check(status: int, call: str):
    if status != RESA_OK:
        raise ResaError(status, call)


def params(keep_ratio: float, n_min_blocks: int, n_local_blocks: int, sm_scale: float = 0.0) -> ResaParamsT:
    return ResaParamsT(float(keep_ratio), int(n_min_blocks), int(n_local_blocks), float(sm_scale), 0)


# ---------------------------------------------------------------- calls ---
def resa_abi_version() -> int:
    return load().resa_abi_version()


def resa_max_selected(cache: ResaCacheT, p: ResaParamsT) -> int:
    n = c_int32(0)
    _check(load().resa_max_selected(ctypes.byref(cache), ctypes.byref(p), ctypes.byref(n)), "resa_max_selected")
    return n.value


def resa_decode_num_splits(cache: ResaCacheT, n_cap: int) -> int:
    s = c_int32(0)
    _check(load().resa_decode_num_splits(ctypes.byref(cache), n_cap, ctypes.byref(s)), "resa_decode_num_splits")
    return s.value


def resa_rectify_num_splits(cache: ResaCacheT, f: int) -> int:
    s = c_int32(0)
    _check(load().resa_rectify_num_splits(ctypes.byref(cache), f, ctypes.byref(s)), "resa_rectify_num_splits")
    return s.value


def resa_set_decode_wait_polls(polls: int = DEFAULT_DECODE_WAIT_POLLS):
    """Polls of one copy barrier after which the sparse decode kernel gives up
    (RESA_DEV_WAIT_TIMEOUT); process-wide. 0 makes every wait give up at once."""
    _check(load().resa_set_decode_wait_polls(int(polls)), "resa_set_decode_wait_polls")


def resa_workspace_size(cache: ResaCacheT, n_cap: int, num_splits: int = 0, max_f: int = 0) -> int:
    n = c_size_t(0)
    _check(load().resa_workspace_size(ctypes.byref(cache), n_cap, num_splits, max_f, ctypes.byref(n)),
           "resa_workspace_size")
    return n.value


def resa_update_summaries(cache: ResaCacheT, block_begin: int = 0, block_end: int = -1, stream=None):
    _check(load().resa_update_summaries(ctypes.byref(cache), block_begin, block_end, _stream(stream)),
           "resa_update_summaries")


def resa_commit_kv(cache: ResaCacheT, k_new, v_new, n_tokens: int, overwrite: bool, stream=None):
    _check(load().resa_commit_kv(ctypes.byref(cache), _ptr(k_new), _ptr(v_new), n_tokens, int(bool(overwrite)),
                                 _stream(stream)), "resa_commit_kv")


def resa_select_blocks(cache: ResaCacheT, q, p: ResaParamsT, indices, counts, n_cap: int, workspace,
                       workspace_bytes: int, stream=None):
    _check(load().resa_select_blocks(ctypes.byref(cache), _ptr(q), ctypes.byref(p), _ptr(indices), _ptr(counts),
                                     n_cap, _ptr(workspace), workspace_bytes, _stream(stream)),
           "resa_select_blocks")


def resa_sparse_decode(cache: ResaCacheT, q, indices, counts, n_cap: int, p: ResaParamsT, out, lse,
                       num_splits: int, workspace, workspace_bytes: int, stream=None):
    _check(load().resa_sparse_decode(ctypes.byref(cache), _ptr(q), _ptr(indices), _ptr(counts), n_cap,
                                     ctypes.byref(p), _ptr(out), _ptr(lse), num_splits, _ptr(workspace),
                                     workspace_bytes, _stream(stream)), "resa_sparse_decode")


def resa_decode_step(cache: ResaCacheT, k_new, v_new, q, p: ResaParamsT, indices, counts, n_cap: int, out, lse,
                     num_splits: int, workspace, workspace_bytes: int, stream=None):
    """One decode step in one call: append (k_new, v_new), select, decode;
    equal to resa_commit_kv + resa_select_blocks + resa_sparse_decode."""
    _check(load().resa_decode_step(ctypes.byref(cache), _ptr(k_new), _ptr(v_new), _ptr(q), ctypes.byref(p),
                                   _ptr(indices), _ptr(counts), n_cap, _ptr(out), _ptr(lse), num_splits,
                                   _ptr(workspace), workspace_bytes, _stream(stream)), "resa_decode_step")


def resa_sparse_decode_static(cache: ResaCacheT, q, indices, counts, n_cap: int, p: ResaParamsT, out, lse,
                              num_splits: int, stream=None):
    """resa_sparse_decode for callers that cannot allocate device memory: no
    workspace argument; the split partials go to the library's static device
    buffer (RESA_STATIC_SCRATCH_BYTES). Calls must not overlap on the GPU."""
    _check(load().resa_sparse_decode_static(ctypes.byref(cache), _ptr(q), _ptr(indices), _ptr(counts), n_cap,
                                            ctypes.byref(p), _ptr(out), _ptr(lse), num_splits, _stream(stream)),
           "resa_sparse_decode_static")


def resa_rectify_attention(cache: ResaCacheT, q_new, k_new, v_new, f: int, p: ResaParamsT, out, lse, workspace,
                           workspace_bytes: int, stream=None):
    _check(load().resa_rectify_attention(ctypes.byref(cache), _ptr(q_new), _ptr(k_new), _ptr(v_new), f,
                                         ctypes.byref(p), _ptr(out), _ptr(lse), _ptr(workspace), workspace_bytes,
                                         _stream(stream)), "resa_rectify_attention")


def resa_read_device_error(cache: ResaCacheT, stream=None) -> tuple[int, int]:
    """(code, detail) of the first device-side error since the last read (0 = none); clears it."""
    code, detail = c_int32(0), c_int32(0)
    st = load().resa_read_device_error(ctypes.byref(cache), ctypes.byref(code), ctypes.byref(detail),
                                       _stream(stream))
    if st not in (RESA_OK, 5):
        raise ResaError(st, "resa_read_device_error")
    return code.value, detail.value


def resa_commit_kv_active(cache: ResaCacheT, active, k_new, v_new, n_tokens: int, overwrite: bool, stream=None):
    """resa_commit_kv for the sequences with active[b] != 0 only (continuous batching)."""
    _check(load().resa_commit_kv_active(ctypes.byref(cache), _ptr(active), _ptr(k_new), _ptr(v_new), n_tokens,
                                        int(bool(overwrite)), _stream(stream)), "resa_commit_kv_active")


def resa_rectify_attention_active(cache: ResaCacheT, active, q_new, k_new, v_new, f: int, p: ResaParamsT, out, lse,
                                  workspace, workspace_bytes: int, stream=None):
    """resa_rectify_attention for the sequences with active[b] != 0 only; the
    output rows of the others are not written."""
    _check(load().resa_rectify_attention_active(ctypes.byref(cache), _ptr(active), _ptr(q_new), _ptr(k_new),
                                                _ptr(v_new), f, ctypes.byref(p), _ptr(out), _ptr(lse),
                                                _ptr(workspace), workspace_bytes, _stream(stream)),
           "resa_rectify_attention_active")


# ------------------------------------------------------ caller buffers ---
class PagedKVCache:
    """Device buffers of one paged cache, owned by torch (caller-side).

    k_pool / v_pool : bf16 [num_pages, Hkv, 16, 128]
    page_table      : int32 [B, max_blocks]
    seq_lens        : int32 [B]
    summaries       : bf16 [B, Hkv, max_blocks, 2, 128]
    device_status   : int32 [4]
    """

    def __init__(self, batch: int, num_q_heads: int, num_kv_heads: int, max_blocks: int, page_table,
                 device="cuda", num_pages: int | None = None, head_dim: int = 128, block_size: int = 16,
                 zero_pools: bool = True):
        import torch
        self.batch, self.Hq, self.Hkv = batch, num_q_heads, num_kv_heads
        self.max_blocks, self.head_dim, self.block_size = max_blocks, head_dim, block_size
        pt = torch.as_tensor(page_table, dtype=torch.int32)
        self.num_pages = int(num_pages if num_pages is not None else int(pt.max()) + 1)
        alloc = torch.zeros if zero_pools else torch.empty
        shape = (self.num_pages, num_kv_heads, block_size, head_dim)
        self.k_pool = alloc(shape, dtype=torch.bfloat16, device=device)
        self.v_pool = alloc(shape, dtype=torch.bfloat16, device=device)
        self.page_table = pt.to(device).contiguous()
        self.seq_lens = torch.zeros(batch, dtype=torch.int32, device=device)
        self.summaries = torch.zeros((batch, num_kv_heads, max_blocks, 2, head_dim), dtype=torch.bfloat16,
                                     device=device)
        self.device_status = torch.zeros(4, dtype=torch.int32, device=device)
        self.struct = ResaCacheT(batch, num_q_heads, num_kv_heads, head_dim, block_size, self.num_pages,
                                 max_blocks, 0, self.k_pool.data_ptr(), self.v_pool.data_ptr(),
                                 self.page_table.data_ptr(), self.seq_lens.data_ptr(), self.summaries.data_ptr(),
                                 self.device_status.data_ptr())

    @property
    def capacity(self) -> int:
        return self.max_blocks * self.block_size
