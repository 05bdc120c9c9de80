"""Drive a decode session of a workload through the C ABI.

Sets up a cache for a ``WorkloadConfig`` (pool sized for the prefix plus
``extra_tokens`` decode steps, page order and reservation order from the
workload), writes each sequence's cached prefix (vision tokens first, then
text) into every layer pool, and runs decode steps: ``kv_begin_step`` then, per
logical layer, ``kv_append`` and ``decode_attention``.  Torch is used only to
hold device buffers and streams.
"""
from __future__ import annotations

import numpy as np

from . import kvdecode as kd
from . import workloads as wl


class DecodeSession:
    def __init__(self, cfg: wl.WorkloadConfig, extra_tokens: int = 8, device="cuda", stream=None,
                 lens=None, slack_pages: int = 8, split_pages: int = 0, host_only: bool = False):
        import torch
        self.torch = torch
        self.cfg = cfg
        self.device = device
        self.stream = stream
        self.lens = np.array(wl.context_lengths(cfg) if lens is None else lens, dtype=np.int64)
        self.lens0 = self.lens.copy()
        P = cfg.page_size
        self.max_pages = int((int(self.lens.max()) + extra_tokens + P - 1) // P)
        self.num_pages = int(sum((int(n) + extra_tokens + P - 1) // P for n in self.lens)) + slack_pages
        flags = kd.KVC_FLAG_HOST_ONLY if host_only else 0
        self.kcfg = kd.make_config(cfg.phys_layers, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim,
                                   self.num_pages, cfg.batch, self.max_pages, page_size=P, flags=flags)
        self.h = kd.kv_cache_create(self.kcfg, stream)
        order = wl.page_order(cfg, self.num_pages)
        if order is not None:
            kd.kv_cache_set_page_order(self.h, order)
        if split_pages:
            kd.kv_cache_set_split_pages(self.h, split_pages)
        self.seq_ids = [kd.kv_seq_create(self.h) for _ in range(cfg.batch)]
        for i, n in wl.reserve_schedule(cfg, self.lens):
            kd.kv_seq_reserve(self.h, self.seq_ids[i], n, stream)

    # ------------------------------------------------------------------ setup
    def fill_prefix(self, layers=None):
        """Write every sequence's cached prefix into the given layer pools."""
        cfg = self.cfg
        layers = range(cfg.phys_layers) if layers is None else layers
        for l in layers:
            for b, seq in enumerate(self.seq_ids):
                n = int(self.lens0[b])
                k = wl.kv_block(cfg, l, b, n, "k", self.device)
                v = wl.kv_block(cfg, l, b, n, "v", self.device)
                kd.kv_write_tokens(self.h, l, seq, 0, n, k, v, self.stream)
                del k, v

    # ------------------------------------------------------------------- step
    def begin_step(self):
        kd.kv_begin_step(self.h, self.seq_ids, self.stream)
        self.lens += 1

    def phys(self, layer: int) -> int:
        return layer % self.cfg.phys_layers

    def append(self, layer: int, k_new, v_new):
        kd.kv_append(self.h, self.phys(layer), self.cfg.batch, k_new, v_new, self.stream)

    def attend(self, layer: int, q, out, scale: float = 0.0):
        kd.decode_attention(self.h, self.phys(layer), self.cfg.batch, q, out, scale, self.stream)

    def append_attend(self, layer: int, q, k_new, v_new, out, scale: float = 0.0):
        """kv_append + decode_attention of one layer in one fused launch."""
        kd.decode_attention_append(self.h, self.phys(layer), self.cfg.batch, q, k_new, v_new, out, scale,
                                   self.stream)

    def query(self, raise_on_device_error=True):
        return kd.kv_cache_query(self.h, raise_on_device_error)

    def close(self):
        if self.h is not None:
            kd.kv_cache_destroy(self.h)
            self.h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
