"""ctypes binding of libkvdecode.so (declared in include/kvdecode.h).

Argument marshalling only: every step of the decode path runs in the CUDA
library.  Functions keep the C names; pointer arguments accept torch tensors
(their ``data_ptr()``), plain integers or None, and ``stream`` accepts a
``torch.cuda.Stream``, a raw handle or None (the legacy default stream).
If the library has not been built, loading fails loudly: there is no
fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libkvdecode.so")

KVC_OK = 0
KVC_ERR_INVALID = -1
KVC_ERR_OOM = -2
KVC_ERR_CUDA = -3
KVC_ERR_PAGE_TABLE = -4
KVC_ERR_UNSUPPORTED = -5
KVC_ERR_DEVICE = -6
KVC_FLAG_HOST_ONLY = 1
KVC_DEVERR_PAGE_RANGE = 1
KVC_DEVERR_WAIT_TIMEOUT = 2
KVC_DEVERR_SEQ_RANGE = 4
KVC_DEVERR_OOM = 8

_NAMES = {KVC_ERR_INVALID: "INVALID", KVC_ERR_OOM: "OOM", KVC_ERR_CUDA: "CUDA",
          KVC_ERR_PAGE_TABLE: "PAGE_TABLE", KVC_ERR_UNSUPPORTED: "UNSUPPORTED",
          KVC_ERR_DEVICE: "DEVICE"}


class KVDecodeError(RuntimeError):
    def __init__(self, code: int, fn: str, msg: str):
        super().__init__(f"{fn} -> KVC_ERR_{_NAMES.get(code, code)}: {msg}")
        self.code = code


class kvc_config(ctypes.Structure):
    _fields_ = [("num_layers", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("max_seqs", ctypes.c_int32),
                ("max_pages_per_seq", ctypes.c_int32), ("flags", ctypes.c_int32),
                ("num_pages", ctypes.c_int64)]


class kvc_stats(ctypes.Structure):
    _fields_ = [("kv_bytes_allocated", ctypes.c_int64), ("pool_bytes", ctypes.c_int64),
                ("pages_in_use", ctypes.c_int64), ("free_pages", ctypes.c_int64),
                ("live_seqs", ctypes.c_int32), ("device_error", ctypes.c_int32),
                ("kernel_launches", ctypes.c_int64)]


_lib = None
_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_SIGS = {
    "kv_cache_create": [ctypes.POINTER(kvc_config), _P, ctypes.POINTER(_P)],
    "kv_cache_destroy": [_P],
    "kv_cache_set_page_order": [_P, _P, _I64],
    "kv_cache_query": [_P, ctypes.POINTER(kvc_stats)],
    "kv_cache_pool": [_P, _I32, ctypes.POINTER(_P), ctypes.POINTER(_P)],
    "kv_cache_set_split_pages": [_P, _I32],
    "kv_seq_create": [_P, ctypes.POINTER(_I32)],
    "kv_seq_reserve": [_P, _I32, _I32, _P],
    "kv_seq_free": [_P, _I32, _P],
    "kv_seq_info": [_P, _I32, ctypes.POINTER(_I32), _P, _I32, ctypes.POINTER(_I32)],
    "kv_write_tokens": [_P, _I32, _I32, _I32, _I32, _P, _P, _P],
    "kv_read_tokens": [_P, _I32, _I32, _I32, _I32, _P, _P, _P],
    "kv_write_varlen": [_P, _I32, _I32, _I32, _P, _P, _P, _P, _P, _P],
    "kv_begin_step": [_P, _I32, _P, _P],
    "kv_append": [_P, _I32, _I32, _P, _P, _P],
    "decode_attention": [_P, _I32, _I32, _P, _P, ctypes.c_float, _P],
    "decode_attention_append": [_P, _I32, _I32, _P, _P, _P, _P, ctypes.c_float, _P],
    "kv_selftest_wait_timeout": [_I64, _P, _P],
    "kv_cache_device_steps": [_P, _I32, _I32, _P],
    "kv_begin_step_device": [_P, _I32, _P, _P],
    "kv_cache_sync": [_P],
    "decode_attention_noalloc": [_P, _P, _I64, _I32, _I32, _I32, _I32, _P, _I32, _P, _P, _P,
                                 ctypes.c_float, _P, _P],
}


def load():
    """Load libkvdecode.so (raises if it is missing)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built; run `python -c \"import __graft_entry__ as g; "
                               f"g.build()\"` (needs nvcc)")
        lib = ctypes.CDLL(LIB_PATH)
        for name, args in _SIGS.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        lib.kv_last_error.argtypes = []
        lib.kv_last_error.restype = ctypes.c_char_p
        _lib = lib
    return _lib


def _ptr(x):
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if isinstance(x, ctypes.Array):
        return ctypes.addressof(x)
    return int(x)


def _stream(s):
    if s is None:
        return None
    if hasattr(s, "cuda_stream"):
        return s.cuda_stream
    return int(s)


def _check(rc: int, fn: str):
    if rc != KVC_OK:
        raise KVDecodeError(rc, fn, load().kv_last_error().decode())


def _i32_array(values):
    vals = [int(v) for v in values]
    return (ctypes.c_int32 * len(vals))(*vals)


# ---------------------------------------------------------------- C names
def kv_cache_create(cfg: kvc_config, stream=None):
    h = _P()
    _check(load().kv_cache_create(ctypes.byref(cfg), _stream(stream), ctypes.byref(h)), "kv_cache_create")
    return h


def kv_cache_destroy(h):
    _check(load().kv_cache_destroy(h), "kv_cache_destroy")


def kv_cache_set_page_order(h, order):
    arr = _i32_array(order)
    _check(load().kv_cache_set_page_order(h, ctypes.addressof(arr), len(arr)), "kv_cache_set_page_order")


def kv_cache_query(h, raise_on_device_error: bool = True) -> kvc_stats:
    s = kvc_stats()
    rc = load().kv_cache_query(h, ctypes.byref(s))
    # A status caused by a device-side error flag still fills the stats.
    if rc != KVC_OK and (raise_on_device_error or s.device_error == 0):
        _check(rc, "kv_cache_query")
    return s


def kv_cache_pool(h, layer: int):
    k, v = _P(), _P()
    _check(load().kv_cache_pool(h, layer, ctypes.byref(k), ctypes.byref(v)), "kv_cache_pool")
    return k.value, v.value


def kv_cache_set_split_pages(h, pages: int):
    _check(load().kv_cache_set_split_pages(h, pages), "kv_cache_set_split_pages")


def kv_seq_create(h) -> int:
    s = _I32()
    _check(load().kv_seq_create(h, ctypes.byref(s)), "kv_seq_create")
    return s.value


def kv_seq_reserve(h, seq: int, n_tokens: int, stream=None):
    _check(load().kv_seq_reserve(h, seq, n_tokens, _stream(stream)), "kv_seq_reserve")


def kv_seq_free(h, seq: int, stream=None):
    _check(load().kv_seq_free(h, seq, _stream(stream)), "kv_seq_free")


def kv_seq_info(h, seq: int):
    """Returns (length, [page ids in logical order])."""
    ln, npg = _I32(), _I32()
    _check(load().kv_seq_info(h, seq, ctypes.byref(ln), None, 0, ctypes.byref(npg)), "kv_seq_info")
    buf = (ctypes.c_int32 * max(1, npg.value))()
    _check(load().kv_seq_info(h, seq, ctypes.byref(ln), ctypes.addressof(buf), npg.value, ctypes.byref(npg)),
           "kv_seq_info")
    return ln.value, list(buf[:npg.value])


def kv_write_tokens(h, layer: int, seq: int, first_pos: int, n: int, k, v, stream=None):
    _check(load().kv_write_tokens(h, layer, seq, first_pos, n, _ptr(k), _ptr(v), _stream(stream)),
           "kv_write_tokens")


def kv_read_tokens(h, layer: int, seq: int, first_pos: int, n: int, k_out, v_out, stream=None):
    _check(load().kv_read_tokens(h, layer, seq, first_pos, n, _ptr(k_out), _ptr(v_out), _stream(stream)),
           "kv_read_tokens")


def kv_write_varlen(h, layer_first: int, n_layers: int, seq_ids, cu_seqlens, k, v, first_pos=None, stream=None):
    """Packed varlen bulk write: block i = rows cu_seqlens[i]..cu_seqlens[i+1]-1
    of k, v ([n_layers][rows][H_kv][d] bf16, device) -> positions
    first_pos[i].. of sequence seq_ids[i] (first_pos None: all 0)."""
    ids = _i32_array(seq_ids)
    cu = _i32_array(cu_seqlens)
    if len(cu) != len(ids) + 1:
        raise ValueError("cu_seqlens needs len(seq_ids) + 1 entries")
    fp = _i32_array(first_pos) if first_pos is not None else None
    if fp is not None and len(fp) != len(ids):
        raise ValueError("first_pos needs len(seq_ids) entries")
    _check(load().kv_write_varlen(h, layer_first, n_layers, len(ids), ctypes.addressof(ids),
                                  ctypes.addressof(fp) if fp is not None else None, ctypes.addressof(cu),
                                  _ptr(k), _ptr(v), _stream(stream)), "kv_write_varlen")


def kv_begin_step(h, seq_ids, stream=None):
    arr = _i32_array(seq_ids)
    _check(load().kv_begin_step(h, len(arr), ctypes.addressof(arr), _stream(stream)), "kv_begin_step")


def kv_append(h, layer: int, batch: int, k_new, v_new, stream=None):
    _check(load().kv_append(h, layer, batch, _ptr(k_new), _ptr(v_new), _stream(stream)), "kv_append")


def decode_attention(h, layer: int, batch: int, q, out, softmax_scale: float = 0.0, stream=None):
    _check(load().decode_attention(h, layer, batch, _ptr(q), _ptr(out), float(softmax_scale), _stream(stream)),
           "decode_attention")


def decode_attention_append(h, layer: int, batch: int, q, k_new, v_new, out, softmax_scale: float = 0.0,
                            stream=None):
    _check(load().decode_attention_append(h, layer, batch, _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(out),
                                          float(softmax_scale), _stream(stream)), "decode_attention_append")


def decode_attention_noalloc(k_pool, v_pool, num_pages: int, num_q_heads: int, num_kv_heads: int,
                             head_dim: int, page_table, max_pages: int, lens, q, out,
                             softmax_scale: float = 0.0, device_error=None, stream=None):
    """Allocation-free decode attention over caller-owned pools and page
    table; ``lens`` is a host sequence of attended token counts, one per row.

    Where torch tensors are passed, their dtype, device, layout and shape are
    checked here before the call, since the kernels read through the raw
    pointers: page_table int32 [len(lens)][max_pages], q and out bf16
    [len(lens)][num_q_heads][head_dim], pools bf16 with at least
    num_pages * num_kv_heads * 16 * head_dim elements, device_error int32."""
    arr = _i32_array(lens)
    batch = len(arr)

    def _tensor(x, name, dtype, shape=None, min_numel=None):
        if not hasattr(x, "data_ptr"):
            return
        if x.dtype != dtype or not x.is_cuda or not x.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA tensor of {dtype}")
        if shape is not None and tuple(x.shape) != tuple(shape):
            raise ValueError(f"{name} must have shape {tuple(shape)}, not {tuple(x.shape)}")
        if min_numel is not None and x.numel() < min_numel:
            raise ValueError(f"{name} holds {x.numel()} elements, fewer than {min_numel}")

    import torch
    _tensor(page_table, "page_table", torch.int32, (batch, max_pages))
    _tensor(q, "q", torch.bfloat16, (batch, num_q_heads, head_dim))
    _tensor(out, "out", torch.bfloat16, (batch, num_q_heads, head_dim))
    pool_elems = int(num_pages) * int(num_kv_heads) * 16 * int(head_dim)
    _tensor(k_pool, "k_pool", torch.bfloat16, min_numel=pool_elems)
    _tensor(v_pool, "v_pool", torch.bfloat16, min_numel=pool_elems)
    _tensor(device_error, "device_error", torch.int32, min_numel=1)
    _check(load().decode_attention_noalloc(_ptr(k_pool), _ptr(v_pool), num_pages, num_q_heads, num_kv_heads,
                                           head_dim, batch, _ptr(page_table), max_pages,
                                           ctypes.addressof(arr), _ptr(q), _ptr(out), float(softmax_scale),
                                           _ptr(device_error), _stream(stream)),
           "decode_attention_noalloc")


def kv_cache_device_steps(h, max_batch: int, enable: bool = True, stream=None):
    _check(load().kv_cache_device_steps(h, max_batch, 1 if enable else 0, _stream(stream)), "kv_cache_device_steps")


def kv_begin_step_device(h, batch: int, seq_ids_dev, stream=None):
    _check(load().kv_begin_step_device(h, batch, _ptr(seq_ids_dev), _stream(stream)), "kv_begin_step_device")


def kv_cache_sync(h):
    _check(load().kv_cache_sync(h), "kv_cache_sync")


def kv_selftest_wait_timeout(limit_ns: int, status, stream=None):
    _check(load().kv_selftest_wait_timeout(int(limit_ns), _ptr(status), _stream(stream)),
           "kv_selftest_wait_timeout")


def make_config(num_layers, num_q_heads, num_kv_heads, head_dim, num_pages, max_seqs, max_pages_per_seq,
                page_size=16, flags=0) -> kvc_config:
    return kvc_config(num_layers=num_layers, num_q_heads=num_q_heads, num_kv_heads=num_kv_heads,
                      head_dim=head_dim, page_size=page_size, max_seqs=max_seqs,
                      max_pages_per_seq=max_pages_per_seq, flags=flags, num_pages=num_pages)
