"""fp64 CPU oracle for paged decode attention and KV append.

TEST INFRASTRUCTURE ONLY.  Nothing in the library's product path imports,
loads or calls this package; only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` do.  It shares no code with the CUDA path:
its C source (``oracle.c``) has its own indexing and its own layout accessor.

Every function here is a thin ctypes wrapper; the arithmetic is in
``oracle.c``, which cites what it follows.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so with gcc (plain C11, -O2, fp64)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math", "-o", tmp, _SRC, "-lm"]
        )
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _bind(lib):
    P = ctypes.c_void_p
    I = ctypes.c_int
    L = ctypes.c_int64
    D = ctypes.c_double
    lib.oracle_append.argtypes = [P, L, L, I, I, I, P, P, P, P, I, I]
    lib.oracle_paged_attention.argtypes = [P, L, L, I, I, I, P, P, P, I, I, I, D, P, I, P]
    lib.oracle_dense_attention.argtypes = [P, P, P, I, I, I, I, D, P]
    lib.oracle_split_attention.argtypes = [P, L, L, I, I, I, P, P, P, I, I, I, D, I, P]
    for f in (lib.oracle_append, lib.oracle_paged_attention, lib.oracle_dense_attention,
              lib.oracle_split_attention):
        f.restype = ctypes.c_int
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
    return _lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def append(pool: np.ndarray, n_pages: int, page_elems: int, bs: int, Hkv: int, d: int,
           k_new, v_new, table, ctx_lens, inplace: bool = False) -> np.ndarray:
    """Return ``pool`` with each sequence's new K/V row written at position
    ctx_len-1 (bit copy); a copy unless ``inplace`` (then ``pool`` must be a
    contiguous uint16 array and is modified)."""
    lib = _load()
    if inplace:
        if pool.dtype != np.uint16 or not pool.flags.c_contiguous:
            raise ValueError("in-place append needs a contiguous uint16 pool")
        out = pool
    else:
        out = np.array(pool, dtype=np.uint16, copy=True)
    table = _c(table, np.int32)
    ctx = _c(ctx_lens, np.int32)
    k_new = _c(k_new, np.uint16)
    v_new = _c(v_new, np.uint16)
    S, max_blocks = table.shape
    rc = lib.oracle_append(_ptr(out), n_pages, page_elems, bs, Hkv, d, _ptr(k_new), _ptr(v_new),
                           _ptr(table), _ptr(ctx), max_blocks, S)
    if rc:
        raise ValueError("oracle_append: index outside the pool or table")
    return out


def paged_attention(pool, n_pages: int, page_elems: int, bs: int, Hkv: int, d: int, q, table,
                    ctx_lens, scale: float, seq_ids=None) -> np.ndarray:
    """fp64 [S, Hq, d] attention output (rows of sequences not in ``seq_ids``
    are NaN when a subset is requested)."""
    lib = _load()
    q = _c(q, np.uint16)
    table = _c(table, np.int32)
    ctx = _c(ctx_lens, np.int32)
    pool = _c(pool, np.uint16)
    S, Hq, _ = q.shape
    max_blocks = table.shape[1]
    out = np.full((S, Hq, d), np.nan, dtype=np.float64)
    ids = None if seq_ids is None else _c(seq_ids, np.int32)
    rc = lib.oracle_paged_attention(_ptr(pool), n_pages, page_elems, bs, Hkv, d, _ptr(q),
                                    _ptr(table), _ptr(ctx), max_blocks, S, Hq, float(scale),
                                    None if ids is None else _ptr(ids),
                                    0 if ids is None else int(ids.size), _ptr(out))
    if rc:
        raise ValueError("oracle_paged_attention: index outside the pool or table")
    return out


def split_attention(pool, n_pages: int, page_elems: int, bs: int, Hkv: int, d: int, q, table,
                    ctx_lens, scale: float, split_len: int) -> np.ndarray:
    """fp64 [S, Hq, d] via per-split partials and the combine step."""
    lib = _load()
    q = _c(q, np.uint16)
    table = _c(table, np.int32)
    ctx = _c(ctx_lens, np.int32)
    pool = _c(pool, np.uint16)
    S, Hq, _ = q.shape
    out = np.zeros((S, Hq, d), dtype=np.float64)
    rc = lib.oracle_split_attention(_ptr(pool), n_pages, page_elems, bs, Hkv, d, _ptr(q),
                                    _ptr(table), _ptr(ctx), table.shape[1], S, Hq, float(scale),
                                    int(split_len), _ptr(out))
    if rc:
        raise ValueError("oracle_split_attention: bad arguments")
    return out


def dense_attention(q, k, v, scale: float) -> np.ndarray:
    """q fp64 [Hq, d]; k, v fp64 [Hkv, n, d] -> fp64 [Hq, d]."""
    lib = _load()
    q = _c(q, np.float64)
    k = _c(k, np.float64)
    v = _c(v, np.float64)
    Hq, d = q.shape
    Hkv, n, _ = k.shape
    out = np.zeros((Hq, d), dtype=np.float64)
    rc = lib.oracle_dense_attention(_ptr(q), _ptr(k), _ptr(v), n, Hq, Hkv, d, float(scale), _ptr(out))
    if rc:
        raise ValueError("oracle_dense_attention: bad arguments")
    return out


def batch_attention(b, pool=None, seq_ids=None) -> np.ndarray:
    """Oracle attention for a ``workloads.Batch`` (after its append)."""
    return paged_attention(b.pool if pool is None else pool, b.n_pages, b.page_elems, b.bs,
                           b.Hkv, b.d, b.q, b.table, b.ctx_lens, b.scale, seq_ids=seq_ids)


def batch_append(b) -> np.ndarray:
    """Oracle pool after the batch's append."""
    return append(b.pool, b.n_pages, b.page_elems, b.bs, b.Hkv, b.d, b.k_new, b.v_new, b.table,
                  b.ctx_lens)


class swapped_library:
    """Context manager: route this module's wrappers through another build of
    the oracle (used by the mutation test to check that the pins fail on a
    deliberately broken copy of oracle.c)."""

    def __init__(self, path: str):
        self.path = path
        self.old = None

    def __enter__(self):
        global _lib
        _load()
        with _lock:
            self.old = _lib
            _lib = _bind(ctypes.CDLL(self.path))
        return self

    def __exit__(self, *exc):
        global _lib
        with _lock:
            _lib = self.old
        return False
