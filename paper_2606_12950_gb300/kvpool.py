"""Thin Python binding of libkvpool's C ABI (include/kvpool.h).

Argument marshalling only: every function has the C name and forwards to the
library; device buffers are passed as raw addresses (ints) or as objects with
``data_ptr()`` (torch tensors), streams as raw handles or objects with
``cuda_stream``.  There is no fallback: if libkvpool.so is missing or fails to
load, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

KV_OK = 0
KV_ERR_INVALID_ARG = -1
KV_ERR_OUT_OF_BLOCKS = -2
KV_ERR_CUDA = -3
KV_ERR_DEVICE_BOUNDS = -4
KV_ERR_UNSUPPORTED = -5
KV_ERR_WORKSPACE = -6
KV_ERR_DEVICE_TIMEOUT = -7
KV_MAX_LAYOUTS = 4

_NAMES = {
    0: "KV_OK", -1: "KV_ERR_INVALID_ARG", -2: "KV_ERR_OUT_OF_BLOCKS", -3: "KV_ERR_CUDA",
    -4: "KV_ERR_DEVICE_BOUNDS", -5: "KV_ERR_UNSUPPORTED", -6: "KV_ERR_WORKSPACE",
    -7: "KV_ERR_DEVICE_TIMEOUT",
}


class KVError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} failed: {_NAMES.get(code, code)}")
        self.code = code


class kv_layout(ctypes.Structure):
    _fields_ = [("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32)]


class kv_pool_desc(ctypes.Structure):
    _fields_ = [
        ("device_base", ctypes.c_void_p),
        ("pool_bytes", ctypes.c_uint64),
        ("block_size", ctypes.c_int32),
        ("num_layouts", ctypes.c_int32),
        ("layouts", kv_layout * KV_MAX_LAYOUTS),
        ("page_bytes", ctypes.c_uint64),
        ("device_error", ctypes.c_void_p),
        ("shuffle_seed", ctypes.c_uint64),
    ]


class kv_seqtab_counters(ctypes.Structure):
    _fields_ = [
        ("blocks_held", ctypes.c_int64),
        ("reserve_calls", ctypes.c_int64),
        ("reservation_misses", ctypes.c_int64),
        ("releases", ctypes.c_int64),
        ("entries_uploaded", ctypes.c_int64),
        ("sync_launches", ctypes.c_int64),
    ]


class kv_stats(ctypes.Structure):
    _fields_ = [
        ("pages_total", ctypes.c_int64),
        ("pages_unassigned", ctypes.c_int64),
        ("blocks_used", ctypes.c_int64 * KV_MAX_LAYOUTS),
        ("blocks_cached", ctypes.c_int64 * KV_MAX_LAYOUTS),
        ("blocks_capacity", ctypes.c_int64 * KV_MAX_LAYOUTS),
        ("bytes_used", ctypes.c_uint64),
        ("bytes_total", ctypes.c_uint64),
        ("bytes_mapped", ctypes.c_uint64),
        ("attn_calls_overlapped", ctypes.c_int64),
    ]


MAP_FN = ctypes.CFUNCTYPE(ctypes.c_int, ctypes.c_void_p, ctypes.c_uint64, ctypes.c_uint64)


class kv_vmm_desc(ctypes.Structure):
    _fields_ = [
        ("chunk_bytes", ctypes.c_uint64),
        ("physical_limit", ctypes.c_uint64),
        ("budget", ctypes.c_void_p),
        ("device", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
        ("map_fn", MAP_FN),
        ("unmap_fn", MAP_FN),
        ("ctx", ctypes.c_void_p),
    ]


class kv_engine(ctypes.Structure):
    _fields_ = [
        ("state", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
        ("ctx_bytes", ctypes.c_uint64),
        ("weight_bytes", ctypes.c_uint64),
        ("kv_bytes", ctypes.c_uint64),
        ("virtual_kv_bytes", ctypes.c_uint64),
        ("weight_reload_s", ctypes.c_double),
        ("ctx_rebuild_s", ctypes.c_double),
        ("kv_swap_in_s", ctypes.c_double),
        ("kv_regen_s", ctypes.c_double),
    ]


class kv_account(ctypes.Structure):
    _fields_ = [
        ("m_res", ctypes.c_uint64),
        ("m_kv", ctypes.c_uint64),
        ("m_kv_virtual", ctypes.c_uint64),
        ("headroom", ctypes.c_int64),
        ("safe", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
        ("overcommit", ctypes.c_double),
    ]


class kv_plan_step(ctypes.Structure):
    _fields_ = [
        ("engine", ctypes.c_int32),
        ("action", ctypes.c_int32),
        ("freed_bytes", ctypes.c_uint64),
        ("cost_s", ctypes.c_double),
    ]


class kv_prefix_group(ctypes.Structure):
    _fields_ = [("count", ctypes.c_int32), ("tokens", ctypes.c_int32)]


class kv_attn_batch(ctypes.Structure):
    _fields_ = [("layout", ctypes.c_int), ("q", ctypes.c_void_p), ("k_new", ctypes.c_void_p),
                ("v_new", ctypes.c_void_p), ("out", ctypes.c_void_p), ("dev_table", ctypes.c_void_p),
                ("dev_ctx_lens", ctypes.c_void_p), ("max_blocks", ctypes.c_int), ("S", ctypes.c_int),
                ("Hq", ctypes.c_int), ("scale", ctypes.c_float), ("workspace", ctypes.c_void_p),
                ("ws_bytes", ctypes.c_size_t)]


KV_ENGINE_IDLE, KV_ENGINE_SLEEPING, KV_ENGINE_SLEEP_PENDING, KV_ENGINE_ACTIVE, KV_ENGINE_COLD = 0, 1, 2, 3, 4
KV_ACT_SLEEP, KV_ACT_EVICT, KV_ACT_STOP, KV_ACT_PREEMPT, KV_ACT_ABORT = 1, 2, 3, 4, 5

_lib = None


def lib() -> ctypes.CDLL:
    """Load libkvpool.so (building it first if its sources are newer)."""
    global _lib
    if _lib is None:
        path = _build.LIB
        if _build.needs_build():
            path = _build.build()
        if not os.path.exists(path):
            raise RuntimeError("libkvpool.so is not built; run paper_2606_12950_gb300.build.build()")
        L = ctypes.CDLL(path)
        P, I, I32, I64, U64, F, SZ = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int32, ctypes.c_int64,
                                       ctypes.c_uint64, ctypes.c_float, ctypes.c_size_t)
        sigs = {
            "kv_pool_create": [ctypes.POINTER(kv_pool_desc), ctypes.POINTER(P)],
            "kv_pool_destroy": [P],
            "kv_alloc_blocks": [P, I, I, P],
            "kv_free_blocks": [P, I, I, P],
            "kv_block_ref": [P, I, I, P],
            "kv_block_refcount": [P, I32, ctypes.POINTER(I32)],
            "kv_pool_stats": [P, ctypes.POINTER(kv_stats)],
            "kv_pool_get_error": [P, P, P],
            "kv_block_table_upload": [P, I, P, I, I, P, P, P, P],
            "kv_append": [P, I, P, P, P, P, I, I, P],
            "kv_workspace_bytes": [P, I, I, I, I, I, ctypes.POINTER(SZ)],
            "kv_workspace_clear": [P, SZ, P],
            "paged_decode_attn": [P, I, P, P, P, P, I, I, I, F, I, P, SZ, P],
            "paged_decode_attn_noalloc": [P, I, P, P, P, P, I, I, I, F, I, P],
            "paged_decode_attn_append": [P, I, P, P, P, P, P, P, I, I, I, F, I, P, SZ, P],
            "paged_decode_attn_seqtab": [P, P, P, P, P, P, P, P, I, I, F, I, P, SZ, P],
            "paged_decode_attn_multi": [P, I, P, P],
            "kv_set_attn_variant": [P, I],
            "kv_set_attn_step_overlap": [P, I],
            "kv_cascade_workspace_bytes": [P, I, I, I, I, ctypes.POINTER(SZ)],
            "kv_pool_create_vmm": [ctypes.POINTER(kv_pool_desc), ctypes.POINTER(kv_vmm_desc), ctypes.POINTER(P)],
            "kv_pool_get_base": [P, ctypes.POINTER(P)],
            "kv_pool_trim": [P, ctypes.POINTER(U64)],
            "kv_budget_create": [U64, ctypes.POINTER(P)],
            "kv_budget_destroy": [P],
            "kv_budget_used": [P, ctypes.POINTER(U64)],
            "paged_decode_attn_cascade": [P, I, P, P, P, P, P, P, I, I, I, F, P, I, P, P, SZ, P],
            "paged_decode_attn_cascade_seqtab": [P, P, P, P, P, P, P, P, I, I, F, P, I, P, P, SZ, P],
            "kv_seqtab_create": [P, I, I, I, ctypes.POINTER(P)],
            "kv_seqtab_destroy": [P],
            "kv_seq_reserve": [P, I, I64],
            "kv_seq_share_prefix": [P, I, I, I],
            "kv_seq_set_len": [P, I, I32],
            "kv_seq_advance": [P, I, P, ctypes.POINTER(I32)],
            "kv_seq_release": [P, I],
            "kv_seq_trim": [P, I],
            "kv_seq_replace": [P, I, P, P, P, P],
            "kv_seqtab_sync": [P, P, P, P],
            "kv_seqtab_host": [P, ctypes.POINTER(P), ctypes.POINTER(P)],
            "kv_seqtab_get_counters": [P, ctypes.POINTER(kv_seqtab_counters)],
            "kv_memory_account": [P, I, U64, U64, U64, ctypes.POINTER(kv_account)],
            "kv_degradation_plan": [P, I, U64, U64, ctypes.c_double, P, I, ctypes.POINTER(I),
                                    ctypes.POINTER(I), ctypes.POINTER(ctypes.c_double),
                                    ctypes.POINTER(U64)],
            "kv_admission_check": [P, I, U64, U64, U64, U64, U64, ctypes.c_double, P, I, ctypes.POINTER(I),
                                   ctypes.POINTER(I), ctypes.POINTER(ctypes.c_double), ctypes.POINTER(I64)],
        }
        for name, args in sigs.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        L.kv_version.argtypes = []
        L.kv_version.restype = ctypes.c_char_p
        _lib = L
    return _lib


def _addr(x) -> int | None:
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return int(x.data_ptr())
    return int(x)


def _stream(s) -> int | None:
    if s is None:
        return None
    if hasattr(s, "cuda_stream"):
        return int(s.cuda_stream)
    return int(s)


def _check(fn: str, rc: int) -> None:
    if rc != KV_OK:
        raise KVError(fn, rc)


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def kv_version() -> str:
    return lib().kv_version().decode()


def kv_pool_create(device_base, pool_bytes: int, block_size: int, layouts, device_error,
                   page_bytes: int = 0, shuffle_seed: int = 0) -> int:
    """Return an opaque pool handle.  ``layouts`` is a list of (Hkv, d)."""
    d = kv_pool_desc()
    d.device_base = _addr(device_base)
    d.pool_bytes = int(pool_bytes)
    d.block_size = int(block_size)
    d.num_layouts = len(layouts)
    for i, (hkv, hd) in enumerate(layouts):
        d.layouts[i] = kv_layout(int(hkv), int(hd))
    d.page_bytes = int(page_bytes)
    d.device_error = _addr(device_error)
    d.shuffle_seed = int(shuffle_seed)
    h = ctypes.c_void_p()
    _check("kv_pool_create", lib().kv_pool_create(ctypes.byref(d), ctypes.byref(h)))
    return h.value


def kv_pool_create_vmm(pool_bytes: int, block_size: int, layouts, device_error, page_bytes: int = 0,
                       shuffle_seed: int = 0, chunk_bytes: int = 0, physical_limit: int = 0, budget=None,
                       device: int = 0, backend=None, device_base=None):
    """A VMM-backed pool.  backend=None: CUDA VMM (the library reserves the
    range); else an object with map(offset, bytes) / unmap(offset, bytes)
    returning 0 on success, over the caller's range device_base."""
    d = kv_pool_desc()
    d.device_base = device_base
    d.pool_bytes = int(pool_bytes)
    d.block_size = int(block_size)
    d.num_layouts = len(layouts)
    for i, (h, hd) in enumerate(layouts):
        d.layouts[i].num_kv_heads = int(h)
        d.layouts[i].head_dim = int(hd)
    d.page_bytes = int(page_bytes)
    d.device_error = _addr(device_error)
    d.shuffle_seed = int(shuffle_seed)
    v = kv_vmm_desc()
    v.chunk_bytes = int(chunk_bytes)
    v.physical_limit = int(physical_limit)
    v.budget = budget
    v.device = int(device)
    keep = None
    if backend is not None:
        keep = (MAP_FN(lambda ctx, off, n: int(backend.map(int(off), int(n)))),
                MAP_FN(lambda ctx, off, n: int(backend.unmap(int(off), int(n)))))
        v.map_fn, v.unmap_fn = keep
    out = ctypes.c_void_p()
    _check("kv_pool_create_vmm", lib().kv_pool_create_vmm(ctypes.byref(d), ctypes.byref(v), ctypes.byref(out)))
    if keep is not None:
        _callbacks[out.value] = keep  # the library keeps calling them until destroy
    return out.value


_callbacks = {}


def kv_pool_get_base(pool) -> int:
    b = ctypes.c_void_p()
    _check("kv_pool_get_base", lib().kv_pool_get_base(pool, ctypes.byref(b)))
    return int(b.value or 0)


def kv_pool_trim(pool) -> int:
    r = ctypes.c_uint64(0)
    _check("kv_pool_trim", lib().kv_pool_trim(pool, ctypes.byref(r)))
    return int(r.value)


def kv_budget_create(limit_bytes: int):
    out = ctypes.c_void_p()
    _check("kv_budget_create", lib().kv_budget_create(int(limit_bytes), ctypes.byref(out)))
    return out.value


def kv_budget_destroy(budget) -> None:
    _check("kv_budget_destroy", lib().kv_budget_destroy(budget))


def kv_budget_used(budget) -> int:
    r = ctypes.c_uint64(0)
    _check("kv_budget_used", lib().kv_budget_used(budget, ctypes.byref(r)))
    return int(r.value)


def kv_pool_destroy(pool) -> None:
    _check("kv_pool_destroy", lib().kv_pool_destroy(pool))
    _callbacks.pop(pool, None)


def kv_alloc_blocks(pool, layout: int, n: int) -> np.ndarray:
    out = np.empty(max(0, int(n)), dtype=np.int32)
    _check("kv_alloc_blocks", lib().kv_alloc_blocks(pool, layout, int(n), out.ctypes.data))
    return out


def kv_free_blocks(pool, layout: int, ids) -> None:
    ids = _i32(ids)
    _check("kv_free_blocks", lib().kv_free_blocks(pool, layout, int(ids.size), ids.ctypes.data))


def kv_block_ref(pool, layout: int, ids) -> None:
    ids = _i32(ids)
    _check("kv_block_ref", lib().kv_block_ref(pool, layout, int(ids.size), ids.ctypes.data))


def kv_block_refcount(pool, block_id: int) -> int:
    c = ctypes.c_int32()
    _check("kv_block_refcount", lib().kv_block_refcount(pool, int(block_id), ctypes.byref(c)))
    return int(c.value)


def kv_pool_stats(pool) -> dict:
    s = kv_stats()
    _check("kv_pool_stats", lib().kv_pool_stats(pool, ctypes.byref(s)))
    return {
        "pages_total": s.pages_total, "pages_unassigned": s.pages_unassigned,
        "blocks_used": list(s.blocks_used), "blocks_cached": list(s.blocks_cached),
        "blocks_capacity": list(s.blocks_capacity), "bytes_used": s.bytes_used,
        "bytes_total": s.bytes_total, "bytes_mapped": s.bytes_mapped,
        "attn_calls_overlapped": s.attn_calls_overlapped,
    }


def kv_pool_get_error(pool, stream, host_buf=None) -> int:
    """Read-and-clear the device error word; synchronises ``stream``'s work
    up to this point when ``host_buf`` (a pinned int32 host tensor) is None."""
    if host_buf is None:
        code = ctypes.c_int32(0)
        _check("kv_pool_get_error", lib().kv_pool_get_error(pool, _stream(stream), ctypes.addressof(code)))
        import torch

        torch.cuda.synchronize()
        return int(code.value)
    _check("kv_pool_get_error", lib().kv_pool_get_error(pool, _stream(stream), _addr(host_buf)))
    return 0


def kv_block_table_upload(pool, layout: int, host_table, host_ctx_lens, dev_table, dev_ctx_lens,
                          stream=None) -> None:
    t = host_table if isinstance(host_table, np.ndarray) and host_table.dtype == np.int32 \
        and host_table.flags.c_contiguous else _i32(host_table)
    lens = _i32(host_ctx_lens)
    S, max_blocks = t.shape
    _check("kv_block_table_upload",
           lib().kv_block_table_upload(pool, layout, t.ctypes.data, int(S), int(max_blocks),
                                       lens.ctypes.data, _addr(dev_table), _addr(dev_ctx_lens),
                                       _stream(stream)))


def kv_append(pool, layout: int, k_new, v_new, dev_table, dev_ctx_lens, max_blocks: int, S: int,
              stream=None) -> None:
    _check("kv_append", lib().kv_append(pool, layout, _addr(k_new), _addr(v_new), _addr(dev_table),
                                        _addr(dev_ctx_lens), int(max_blocks), int(S), _stream(stream)))


def kv_workspace_bytes(pool, layout: int, S: int, Hq: int, max_blocks: int, num_splits: int = 0) -> int:
    n = ctypes.c_size_t(0)
    _check("kv_workspace_bytes", lib().kv_workspace_bytes(pool, layout, int(S), int(Hq), int(max_blocks),
                                                          int(num_splits), ctypes.byref(n)))
    return int(n.value)


def kv_workspace_clear(workspace, ws_bytes: int, stream=None) -> None:
    _check("kv_workspace_clear", lib().kv_workspace_clear(_addr(workspace), int(ws_bytes), _stream(stream)))


def paged_decode_attn(pool, layout: int, q, out, dev_table, dev_ctx_lens, max_blocks: int, S: int,
                      Hq: int, scale: float, num_splits: int, workspace, ws_bytes: int,
                      stream=None) -> None:
    _check("paged_decode_attn",
           lib().paged_decode_attn(pool, layout, _addr(q), _addr(out), _addr(dev_table),
                                   _addr(dev_ctx_lens), int(max_blocks), int(S), int(Hq), float(scale),
                                   int(num_splits), _addr(workspace), int(ws_bytes), _stream(stream)))


def paged_decode_attn_append(pool, layout: int, q, k_new, v_new, out, dev_table, dev_ctx_lens, max_blocks: int,
                             S: int, Hq: int, scale: float, num_splits: int, workspace, ws_bytes: int,
                             stream=None) -> None:
    """kv_append + paged_decode_attn fused into one pass."""
    _check("paged_decode_attn_append",
           lib().paged_decode_attn_append(pool, layout, _addr(q), _addr(k_new), _addr(v_new), _addr(out),
                                          _addr(dev_table), _addr(dev_ctx_lens), int(max_blocks), int(S),
                                          int(Hq), float(scale), int(num_splits), _addr(workspace),
                                          int(ws_bytes), _stream(stream)))


def paged_decode_attn_seqtab(pool, seqtab, q, k_new, v_new, out, dev_table, dev_ctx_lens, S: int, Hq: int,
                             scale: float, num_splits: int, workspace, ws_bytes: int, stream=None) -> None:
    """kv_seqtab_sync + paged_decode_attn(_append) in one launch when the
    table's lengths and changed entries fit the decode kernel's parameters."""
    h = seqtab.handle if isinstance(seqtab, SeqTab) else seqtab
    _check("paged_decode_attn_seqtab",
           lib().paged_decode_attn_seqtab(pool, h, _addr(q), _addr(k_new), _addr(v_new), _addr(out),
                                          _addr(dev_table), _addr(dev_ctx_lens), int(S), int(Hq), float(scale),
                                          int(num_splits), _addr(workspace), int(ws_bytes), _stream(stream)))


def attn_batches(batches) -> "ctypes.Array":
    """kv_attn_batch array from dicts with the struct's fields (tensors or
    addresses for the pointers; k_new / v_new None for no append)."""
    arr = (kv_attn_batch * max(1, len(batches)))()
    for i, b in enumerate(batches):
        arr[i] = kv_attn_batch(int(b["layout"]), _addr(b["q"]), _addr(b.get("k_new")), _addr(b.get("v_new")),
                               _addr(b["out"]), _addr(b["dev_table"]), _addr(b["dev_ctx_lens"]),
                               int(b["max_blocks"]), int(b["S"]), int(b["Hq"]), float(b["scale"]),
                               _addr(b["workspace"]), int(b["ws_bytes"]))
    return arr


def paged_decode_attn_multi(pool, batches, stream=None) -> None:
    """Several batches (co-located layouts) in one call; `batches` is a
    kv_attn_batch array (attn_batches) or a list of dicts."""
    arr = batches if isinstance(batches, ctypes.Array) else attn_batches(batches)
    n = len(batches)
    _check("paged_decode_attn_multi", lib().paged_decode_attn_multi(pool, n, ctypes.addressof(arr), _stream(stream)))


def paged_decode_attn_noalloc(pool, layout: int, q, out, dev_table, dev_ctx_lens, max_blocks: int, S: int,
                              Hq: int, scale: float, num_splits: int = 0, stream=None) -> None:
    """paged_decode_attn with the library's fixed 32 MiB scratch instead of a
    caller workspace (for callers that cannot allocate)."""
    _check("paged_decode_attn_noalloc",
           lib().paged_decode_attn_noalloc(pool, layout, _addr(q), _addr(out), _addr(dev_table),
                                           _addr(dev_ctx_lens), int(max_blocks), int(S), int(Hq), float(scale),
                                           int(num_splits), _stream(stream)))


class PrefixPlan:
    """Groups of sequences sharing a prefix: [(members, tokens), ...],
    marshalled once for paged_decode_attn_cascade."""

    def __init__(self, groups):
        groups = [(list(map(int, m)), int(t)) for m, t in groups]
        self.n_groups = len(groups)
        self.groups = (kv_prefix_group * max(1, self.n_groups))()
        members = [s for m, _ in groups for s in m]
        self.members = (ctypes.c_int32 * max(1, len(members)))(*members)
        for i, (m, t) in enumerate(groups):
            self.groups[i].count = len(m)
            self.groups[i].tokens = t
        self.n_members = len(members)


def kv_cascade_workspace_bytes(pool, layout: int, S: int, Hq: int, max_blocks: int) -> int:
    n = ctypes.c_size_t(0)
    _check("kv_cascade_workspace_bytes", lib().kv_cascade_workspace_bytes(pool, layout, int(S), int(Hq),
                                                                          int(max_blocks), ctypes.byref(n)))
    return int(n.value)


def paged_decode_attn_cascade(pool, layout: int, q, k_new, v_new, out, dev_table, dev_ctx_lens, max_blocks: int,
                              S: int, Hq: int, scale: float, plan: PrefixPlan, workspace, ws_bytes: int,
                              stream=None) -> None:
    _check("paged_decode_attn_cascade",
           lib().paged_decode_attn_cascade(pool, layout, _addr(q), _addr(k_new), _addr(v_new), _addr(out),
                                           _addr(dev_table), _addr(dev_ctx_lens), int(max_blocks), int(S), int(Hq),
                                           float(scale), ctypes.addressof(plan.groups), plan.n_groups,
                                           ctypes.addressof(plan.members), _addr(workspace), int(ws_bytes),
                                           _stream(stream)))


def paged_decode_attn_cascade_seqtab(pool, seqtab, q, k_new, v_new, out, dev_table, dev_ctx_lens, S: int,
                                     Hq: int, scale: float, plan: PrefixPlan, workspace, ws_bytes: int,
                                     stream=None) -> None:
    """kv_seqtab_sync + paged_decode_attn_cascade, the sync carried by the
    kernel that writes the plan when it fits there."""
    h = seqtab.handle if isinstance(seqtab, SeqTab) else seqtab
    _check("paged_decode_attn_cascade_seqtab",
           lib().paged_decode_attn_cascade_seqtab(pool, h, _addr(q), _addr(k_new), _addr(v_new), _addr(out),
                                                  _addr(dev_table), _addr(dev_ctx_lens), int(S), int(Hq),
                                                  float(scale), ctypes.addressof(plan.groups), plan.n_groups,
                                                  ctypes.addressof(plan.members), _addr(workspace), int(ws_bytes),
                                                  _stream(stream)))


def kv_set_attn_variant(pool, variant: int) -> None:
    _check("kv_set_attn_variant", lib().kv_set_attn_variant(pool, int(variant)))


def kv_set_attn_step_overlap(pool, on: bool) -> None:
    """Let a decode kernel start while the previous attention call's combine
    on the same stream finishes (see kvpool.h)."""
    _check("kv_set_attn_step_overlap", lib().kv_set_attn_step_overlap(pool, int(bool(on))))


# ------------------------------------------------------------ sequence tables
class SeqTab:
    """Handle of a host sequence table (kv_seqtab_*)."""

    def __init__(self, pool, layout: int, max_seqs: int, max_blocks: int):
        h = ctypes.c_void_p()
        _check("kv_seqtab_create", lib().kv_seqtab_create(pool, layout, int(max_seqs), int(max_blocks),
                                                          ctypes.byref(h)))
        self.handle = h.value
        self.S = int(max_seqs)
        self.max_blocks = int(max_blocks)
        self._lens_view = None

    def close(self) -> None:
        if self.handle:
            self._lens_view = None
            _check("kv_seqtab_destroy", lib().kv_seqtab_destroy(self.handle))
            self.handle = None

    def reserve(self, s: int, tokens: int) -> None:
        _check("kv_seq_reserve", lib().kv_seq_reserve(self.handle, int(s), int(tokens)))

    def share_prefix(self, dst: int, src: int, nblocks: int) -> None:
        _check("kv_seq_share_prefix", lib().kv_seq_share_prefix(self.handle, int(dst), int(src), int(nblocks)))

    def set_len(self, s: int, length: int) -> None:
        _check("kv_seq_set_len", lib().kv_seq_set_len(self.handle, int(s), int(length)))

    def advance(self, seqs=None) -> int:
        g = ctypes.c_int32(0)
        if seqs is None:
            _check("kv_seq_advance", lib().kv_seq_advance(self.handle, 0, None, ctypes.byref(g)))
        else:
            a = _i32(seqs)
            _check("kv_seq_advance", lib().kv_seq_advance(self.handle, int(a.size), a.ctypes.data, ctypes.byref(g)))
        return int(g.value)

    def release(self, s: int) -> None:
        _check("kv_seq_release", lib().kv_seq_release(self.handle, int(s)))

    def trim(self, s: int) -> None:
        _check("kv_seq_trim", lib().kv_seq_trim(self.handle, int(s)))

    def replace(self, slots, reserve_tokens, lens) -> np.ndarray:
        """Release each listed slot, then reserve and set the length of its
        new sequence, in order (kv_seq_replace).  Returns the per-slot status:
        0, or KV_ERR_OUT_OF_BLOCKS where that admission found the pool full
        (the slot is left empty)."""
        a = _i32(slots)
        r = np.ascontiguousarray(reserve_tokens, dtype=np.int64)
        n = _i32(lens)
        if not (a.shape == r.shape == n.shape and a.ndim == 1):
            raise ValueError("slots, reserve_tokens and lens must be 1-D and of one length")
        st = np.zeros(a.size, dtype=np.int32)
        _check("kv_seq_replace", lib().kv_seq_replace(self.handle, int(a.size), a.ctypes.data, r.ctypes.data,
                                                      n.ctypes.data, st.ctypes.data))
        return st

    def sync(self, dev_table, dev_ctx_lens, stream=None) -> None:
        _check("kv_seqtab_sync", lib().kv_seqtab_sync(self.handle, _addr(dev_table), _addr(dev_ctx_lens),
                                                      _stream(stream)))

    def host(self):
        """Copies of the host table [S, max_blocks] and lengths [S]."""
        t = ctypes.c_void_p()
        l = ctypes.c_void_p()
        _check("kv_seqtab_host", lib().kv_seqtab_host(self.handle, ctypes.byref(t), ctypes.byref(l)))
        tab = np.ctypeslib.as_array(ctypes.cast(t, ctypes.POINTER(ctypes.c_int32)), shape=(self.S * self.max_blocks,))
        lens = np.ctypeslib.as_array(ctypes.cast(l, ctypes.POINTER(ctypes.c_int32)), shape=(self.S,))
        return tab.reshape(self.S, self.max_blocks).copy(), lens.copy()

    def lens(self) -> np.ndarray:
        """Copy of the host lengths only."""
        if self.handle is None:
            raise KVError("kv_seqtab_host", KV_ERR_INVALID_ARG)
        if self._lens_view is None:
            # the table's length array keeps its address for the table's life;
            # the view is dropped when the table closes
            t = ctypes.c_void_p()
            l = ctypes.c_void_p()
            _check("kv_seqtab_host", lib().kv_seqtab_host(self.handle, ctypes.byref(t), ctypes.byref(l)))
            self._lens_view = np.ctypeslib.as_array(ctypes.cast(l, ctypes.POINTER(ctypes.c_int32)), shape=(self.S,))
        return self._lens_view.copy()

    def counters(self) -> dict:
        c = kv_seqtab_counters()
        _check("kv_seqtab_get_counters", lib().kv_seqtab_get_counters(self.handle, ctypes.byref(c)))
        return {f: getattr(c, f) for f, _ in kv_seqtab_counters._fields_}

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _engines(engines):
    """A sequence of kv_engine or of dicts with kv_engine's field names."""
    arr = (kv_engine * max(1, len(engines)))()
    for i, e in enumerate(engines):
        if isinstance(e, kv_engine):
            arr[i] = e
        else:
            for k, v in e.items():
                setattr(arr[i], k, v)
    return arr


def _steps(arr, n):
    return [{"engine": arr[i].engine, "action": arr[i].action, "freed_bytes": arr[i].freed_bytes,
             "cost_s": arr[i].cost_s} for i in range(n)]


def kv_memory_account(engines, m_total: int, m_other: int, extra_kv_bytes: int = 0) -> dict:
    arr = _engines(engines)
    out = kv_account()
    _check("kv_memory_account", lib().kv_memory_account(ctypes.addressof(arr), len(engines), m_total, m_other,
                                                        extra_kv_bytes, ctypes.byref(out)))
    return {"m_res": out.m_res, "m_kv": out.m_kv, "m_kv_virtual": out.m_kv_virtual, "headroom": out.headroom,
            "safe": bool(out.safe), "overcommit": out.overcommit}


def kv_degradation_plan(engines, required: int, host_swap_bytes: int = 0, c_int: float = 0.0) -> dict:
    """Alg. 2 + Eq. 3.  Returns {ok, steps, interrupt, c_deg, freed}; ok is False
    when the plan cannot free `required` (KV_ERR_OUT_OF_BLOCKS)."""
    arr = _engines(engines)
    cap = max(1, len(engines))
    steps = (kv_plan_step * cap)()
    n, intr, c, fr = ctypes.c_int(), ctypes.c_int(), ctypes.c_double(), ctypes.c_uint64()
    rc = lib().kv_degradation_plan(ctypes.addressof(arr), len(engines), required, host_swap_bytes, c_int,
                                   ctypes.addressof(steps), cap, ctypes.byref(n), ctypes.byref(intr),
                                   ctypes.byref(c), ctypes.byref(fr))
    if rc not in (KV_OK, KV_ERR_OUT_OF_BLOCKS):
        raise KVError("kv_degradation_plan", rc)
    return {"ok": rc == KV_OK, "steps": _steps(steps, n.value), "interrupt": bool(intr.value), "c_deg": c.value,
            "freed": fr.value}


def kv_admission_check(engines, m_total: int, m_other: int, extra_kv_bytes: int, demand: int,
                       host_swap_bytes: int = 0, c_int: float = 0.0) -> dict:
    """§III-C admission.  Returns {ok, steps, interrupt, c_deg, headroom}."""
    arr = _engines(engines)
    cap = max(1, len(engines))
    steps = (kv_plan_step * cap)()
    n, intr, c, h = ctypes.c_int(), ctypes.c_int(), ctypes.c_double(), ctypes.c_int64()
    rc = lib().kv_admission_check(ctypes.addressof(arr), len(engines), m_total, m_other, extra_kv_bytes, demand,
                                  host_swap_bytes, c_int, ctypes.addressof(steps), cap, ctypes.byref(n),
                                  ctypes.byref(intr), ctypes.byref(c), ctypes.byref(h))
    if rc not in (KV_OK, KV_ERR_OUT_OF_BLOCKS):
        raise KVError("kv_admission_check", rc)
    return {"ok": rc == KV_OK, "steps": _steps(steps, n.value), "interrupt": bool(intr.value), "c_deg": c.value,
            "headroom": h.value}
