"""Float64 CPU oracle for paged decode attention (HeteroServe language decoding).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` leg (and ``--impl reference`` arm) of ``bench.py`` may import
this package.  The product path (``paper_2603_12707_gb300``) never imports,
links or runs anything here, and nothing here imports the product.

Contents
--------
* ``decode_oracle.c`` -- the definition of one decode step of attention over
  a KV cache of ``N_v + s_text`` tokens (Sec. 4.1 Eq. 1 for what the cache holds,
  Sec. 2 / Sec. 5.1 for decode streaming it, MHA and GQA backends), in float64,
  plus the paged scatter / gather that define kv_append and the prefix write.
* ``allocator_model.py`` -- the lazy page allocation policy (Sec. 5.4 "Lazy KV
  Cache Allocation") as a plain Python model.
* ``footprint.py`` -- Eq. 1, ``D_KV = 2 L n_kv d_h s_ctx b``.

Pins: ``tests/test_oracle_pins.py`` checks every function here against closed
forms, library routines and brute force, never against itself.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

from .allocator_model import PagePoolModel, OutOfPages  # noqa: F401
from .footprint import kv_bytes_eq1, kv_bytes_paged  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "decode_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``decode_oracle.c`` into ``liboracle.so`` (gcc, OpenMP)."""
    stale = (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11",
               "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            lib.oracle_bf16_to_f64.argtypes = [P, P, i64]
            lib.oracle_bf16_to_f64.restype = None
            lib.oracle_decode_attention.argtypes = [i32, i32, i32, i32, P, P, P, P, f64, P, P]
            lib.oracle_decode_attention.restype = ctypes.c_int
            lib.oracle_kv_gather.argtypes = [P, i64, i32, i32, i32, P, i64, i64, P]
            lib.oracle_kv_gather.restype = ctypes.c_int
            lib.oracle_kv_scatter.argtypes = [P, i64, i32, i32, i32, P, i64, i64, P]
            lib.oracle_kv_scatter.restype = ctypes.c_int
            lib.oracle_decode_attention_paged.argtypes = [
                i32, i32, i32, i32, i32, P, P, P, i32, P, P, i64, f64, P]
            lib.oracle_decode_attention_paged.restype = ctypes.c_int
            _lib = lib
    return _lib


def _u16(a) -> np.ndarray:
    """bf16 bit patterns as a C-contiguous uint16 array (accepts uint16/int16
    numpy arrays or CPU torch bf16 tensors)."""
    if hasattr(a, "view") and hasattr(a, "dtype") and str(getattr(a, "dtype", "")) == "torch.bfloat16":
        import torch  # local: only for the conversion of caller tensors
        a = a.detach().cpu().contiguous().view(torch.int16).numpy()
    a = np.ascontiguousarray(a)
    if a.dtype == np.int16:
        a = a.view(np.uint16)
    if a.dtype != np.uint16:
        raise TypeError(f"expected bf16 bit patterns (uint16), got {a.dtype}")
    return a


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def bf16_to_f64(bits) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    b = _u16(bits)
    out = np.empty(b.shape, dtype=np.float64)
    _load().oracle_bf16_to_f64(_ptr(b), _ptr(out), b.size)
    return out


def decode_attention(q, kv_lens, k, v, scale: float | None = None, return_wsum: bool = False):
    """Decode attention over logical-order K/V.

    q: [B, H_q, d] bf16 bits; kv_lens: [B] token counts (>= 1);
    k, v: [sum(kv_lens), H_kv, d] bf16 bits, sequences concatenated in batch
    order, each in logical token order.  Returns float64 [B, H_q, d]
    (and the per-head softmax weight sums when ``return_wsum``).
    """
    q, k, v = _u16(q), _u16(k), _u16(v)
    B, H_q, d = q.shape
    H_kv = k.shape[1]
    lens = np.asarray(kv_lens, dtype=np.int64)
    off = np.zeros(B + 1, dtype=np.int64)
    off[1:] = np.cumsum(lens)
    if k.shape != (off[-1], H_kv, d) or v.shape != k.shape:
        raise ValueError("k/v shape does not match kv_lens")
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    out = np.empty((B, H_q, d), dtype=np.float64)
    ws = np.empty((B, H_q), dtype=np.float64)
    rc = _load().oracle_decode_attention(B, H_q, H_kv, d, _ptr(q), _ptr(off), _ptr(k), _ptr(v),
                                         float(scale), _ptr(out), _ptr(ws))
    if rc != 0:
        raise ValueError("oracle_decode_attention rejected its inputs")
    return (out, ws) if return_wsum else out


def kv_scatter(pool, page_table_row, first: int, src, page_size: int):
    """Write src [n, H_kv, d] into logical positions [first, first+n) of a
    [num_pages, H_kv, P, d] pool (in place)."""
    if pool.dtype != np.uint16 or not pool.flags.c_contiguous:
        raise TypeError("pool must be a C-contiguous uint16 array")
    src = _u16(src)
    row = np.ascontiguousarray(page_table_row, dtype=np.int32)
    num_pages, H_kv, P, d = pool.shape
    if P != page_size:
        raise ValueError("page size mismatch")
    rc = _load().oracle_kv_scatter(_ptr(pool), num_pages, H_kv, P, d, _ptr(row), first,
                                   src.shape[0], _ptr(src))
    if rc != 0:
        raise ValueError("page id outside the pool")


def kv_gather(pool, page_table_row, first: int, n: int) -> np.ndarray:
    """Read logical positions [first, first+n) of one sequence -> [n, H_kv, d]."""
    pool = _u16(pool)
    row = np.ascontiguousarray(page_table_row, dtype=np.int32)
    num_pages, H_kv, P, d = pool.shape
    dst = np.empty((n, H_kv, d), dtype=np.uint16)
    rc = _load().oracle_kv_gather(_ptr(pool), num_pages, H_kv, P, d, _ptr(row), first, n,
                                  _ptr(dst))
    if rc != 0:
        raise ValueError("page id outside the pool")
    return dst


def decode_attention_paged(q, lens, page_table, k_pool, v_pool, scale: float | None = None):
    """Decode attention reading K/V through the oracle's own page-table walk.

    q [B, H_q, d]; lens [B]; page_table [B, max_pages] int32;
    k_pool, v_pool [num_pages, H_kv, P, d] bf16 bits.
    """
    q, k_pool, v_pool = _u16(q), _u16(k_pool), _u16(v_pool)
    B, H_q, d = q.shape
    num_pages, H_kv, P, d2 = k_pool.shape
    if d2 != d or v_pool.shape != k_pool.shape:
        raise ValueError("pool shape mismatch")
    lens = np.ascontiguousarray(lens, dtype=np.int32)
    pt = np.ascontiguousarray(page_table, dtype=np.int32)
    if scale is None:
        scale = 1.0 / np.sqrt(d)
    out = np.empty((B, H_q, d), dtype=np.float64)
    rc = _load().oracle_decode_attention_paged(B, H_q, H_kv, d, P, _ptr(q), _ptr(lens), _ptr(pt),
                                               pt.shape[1], _ptr(k_pool), _ptr(v_pool), num_pages,
                                               float(scale), _ptr(out))
    if rc != 0:
        raise ValueError("oracle_decode_attention_paged rejected its inputs")
    return out
