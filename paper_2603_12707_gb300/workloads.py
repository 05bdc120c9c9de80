"""Seeded synthetic workloads for paged decode attention.

This module only draws inputs: shapes, context lengths, page orders and bf16
values.  It holds none of the attention arithmetic, and both the CUDA path
(tests, bench) and the float64 oracle consume what it draws.

The shapes follow the two models the paper serves: LLaVA-1.5-7B (MHA, 32
layers, 32 KV heads, d_h = 128, fixed 576 vision tokens) and Qwen2.5-VL-7B
(GQA, 28 layers, 28 query / 4 KV heads, dynamic-resolution vision prefix)
(Sec. 6.1 "Models"; Sec. 4.2 Table 3 and "Handling dynamic visual token counts").
The paper's own workload (COCO 2017 val images, one prompt, up to 128 output
tokens, Sec. 6.1 "Workload") is not available here; these seeded draws stand in
for it.  Recipe:

* integers (lengths, vision-prefix sizes, page permutations): numpy PCG64
  seeded with ``seed``;
* values: ``torch.randn`` (float32) from a ``torch.Generator`` on the target
  device seeded per (layer, sequence, K/V) or per (step, layer, tensor), times
  the config's scale, rounded to bf16 (round to nearest even).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import numpy as np


@dataclasses.dataclass(frozen=True)
class WorkloadConfig:
    name: str
    num_layers: int            # logical layers attended per decode step
    phys_layers: int           # layer pools actually allocated (logical l -> l % phys)
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    batch: int
    page_size: int
    seed: int
    kv_scale: float            # K and V are N(0,1) * kv_scale
    q_scale: float             # Q is N(0,1) * q_scale
    ctx_kind: str              # how cached lengths are drawn (see context_lengths)
    page_order: str            # "sequential" | "shuffled" | "interleaved"
    description: str

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads


CONFIGS = {
    "tiny": WorkloadConfig(
        "tiny", 1, 1, 8, 8, 64, 4, 16, 1000, 1.0, 1.0, "tiny", "shuffled",
        "tiny MHA decode: 1 layer, 8/8 heads, d 64, batch 4, 64 vision + 32 text tokens, "
        "page 16, N(0,1) Q/K/V, random page permutation"),
    "llava": WorkloadConfig(
        "llava", 32, 32, 32, 32, 128, 64, 16, 1001, 1.0 / math.sqrt(128.0), 1.0, "llava", "shuffled",
        "LLaVA-1.5-7B-shaped decode: 32 layers, 32/32 heads (MHA), d 128, batch 64, "
        "576 vision + U[64,512] prompt + U{0..256} generated tokens, page 16, "
        "KV N(0,1)/sqrt(128), shuffled page table"),
    "qwen": WorkloadConfig(
        "qwen", 28, 28, 28, 4, 128, 32, 16, 1002, 1.0, 1.0, "qwen", "sequential",
        "Qwen2.5-VL-7B-shaped GQA decode: 28 layers, 28/4 heads (group 7), d 128, batch 32, "
        "N_v uniform over {256,576,1024,2048,4096} + U[32,512] prompt, page 16, KV N(0,1)"),
    "ragged": WorkloadConfig(
        "ragged", 32, 8, 32, 32, 128, 256, 16, 1003, 1.0, 1.0, "ragged", "interleaved",
        "ragged mixed batch: 256 LLaVA-shaped requests (32/32 heads, d 128, 32 layers backed by "
        "8 layer pools), total context log-uniform in [600,8192] with a 576-token vision prefix, "
        "pages allocated interleaved across requests, KV N(0,1)"),
    "long": WorkloadConfig(
        "long", 28, 28, 28, 4, 128, 8, 16, 1004, 1.0, 1.0, "long", "sequential",
        "long multi-image context: Qwen2.5-VL-7B GQA shape (28/4 heads, d 128, 28 layers), "
        "batch 8, 32768 tokens (8 images x 2048 vision + 16384 text), page 16, KV N(0,1)"),
}

QWEN_NV_CHOICES = (256, 576, 1024, 2048, 4096)


def custom(name="custom", num_layers=1, num_q_heads=8, num_kv_heads=8, head_dim=64, batch=4,
           page_size=16, seed=7, kv_scale=1.0, q_scale=1.0, lens=None, page_order="shuffled",
           phys_layers=None) -> WorkloadConfig:
    """A small config for tests; ``lens`` (cached tokens per sequence) is
    carried in the name-independent ``ctx_kind`` field as 'fixed:<csv>'."""
    kind = "fixed:" + ",".join(str(int(x)) for x in lens) if lens is not None else "tiny"
    return WorkloadConfig(name, num_layers, phys_layers or num_layers, num_q_heads, num_kv_heads,
                          head_dim, batch, page_size, seed, kv_scale, q_scale, kind, page_order,
                          "test config")


def _rng(cfg: WorkloadConfig, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([cfg.seed, stream]))


def vision_prefix_lengths(cfg: WorkloadConfig) -> np.ndarray:
    """N_v per sequence (the first N_v cached positions hold the vision KV)."""
    B = cfg.batch
    if cfg.ctx_kind == "tiny":
        return np.full(B, 64, dtype=np.int64)
    if cfg.ctx_kind in ("llava", "ragged"):
        return np.full(B, 576, dtype=np.int64)
    if cfg.ctx_kind == "qwen":
        return _rng(cfg, 1).choice(np.array(QWEN_NV_CHOICES, dtype=np.int64), size=B)
    if cfg.ctx_kind == "long":
        return np.full(B, 8 * 2048, dtype=np.int64)
    if cfg.ctx_kind.startswith("fixed:"):
        lens = context_lengths(cfg)
        return np.minimum(lens, 64)
    raise ValueError(cfg.ctx_kind)


def context_lengths(cfg: WorkloadConfig) -> np.ndarray:
    """Tokens cached per sequence before the decode step (s_b)."""
    B = cfg.batch
    if cfg.ctx_kind == "tiny":
        return np.full(B, 64 + 32, dtype=np.int64)
    if cfg.ctx_kind == "llava":
        r = _rng(cfg, 2)
        prompt = r.integers(64, 512, size=B, endpoint=True)
        generated = r.integers(0, 256, size=B, endpoint=True)
        return 576 + prompt + generated
    if cfg.ctx_kind == "qwen":
        prompt = _rng(cfg, 2).integers(32, 512, size=B, endpoint=True)
        return vision_prefix_lengths(cfg) + prompt
    if cfg.ctx_kind == "ragged":
        u = _rng(cfg, 2).random(B)
        total = np.exp(np.log(600.0) + u * (np.log(8192.0) - np.log(600.0)))
        return np.clip(np.rint(total).astype(np.int64), 600, 8192)
    if cfg.ctx_kind == "long":
        return np.full(B, 32768, dtype=np.int64)
    if cfg.ctx_kind.startswith("fixed:"):
        lens = np.array([int(x) for x in cfg.ctx_kind[6:].split(",")], dtype=np.int64)
        if lens.size != B:
            raise ValueError("fixed lengths do not match the batch")
        return lens
    raise ValueError(cfg.ctx_kind)


def pages_for(lens, page_size: int) -> int:
    return int(sum((int(n) + page_size - 1) // page_size for n in lens))


def page_order(cfg: WorkloadConfig, num_pages: int) -> Optional[np.ndarray]:
    """Pop order to install in the allocator before any sequence is created:
    a seeded permutation for "shuffled", None (identity) otherwise."""
    if cfg.page_order == "shuffled":
        return _rng(cfg, 3).permutation(num_pages).astype(np.int32)
    return None


def reserve_schedule(cfg: WorkloadConfig, lens) -> list:
    """Ordered (sequence index, tokens) reservations that build the prefix.

    "interleaved" hands out pages round-robin across requests (one page worth
    of tokens per request per round), which fragments every page table; the
    other orders reserve each sequence's whole context at once.
    """
    lens = [int(n) for n in lens]
    if cfg.page_order != "interleaved":
        return [(i, n) for i, n in enumerate(lens)]
    P = cfg.page_size
    done = [0] * len(lens)
    out = []
    while True:
        progressed = False
        for i, n in enumerate(lens):
            if done[i] < n:
                take = min(P, n - done[i])
                out.append((i, take))
                done[i] += take
                progressed = True
        if not progressed:
            return out


def _gen(device, seed: int):
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFFFFFF)
    return g


def _draw(shape, scale: float, seed: int, device):
    import torch
    g = _gen(device, seed)
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if scale != 1.0:
        x = x * scale
    return x.to(torch.bfloat16)


def _mix(*parts: int) -> int:
    """Deterministic 63-bit seed from integers (splitmix64 finaliser)."""
    h = 0x9E3779B97F4A7C15
    for p in parts:
        h ^= (int(p) + 0x9E3779B97F4A7C15 + ((h << 6) & 0xFFFFFFFFFFFFFFFF) + (h >> 2)) & 0xFFFFFFFFFFFFFFFF
        h = (h ^ (h >> 30)) * 0xBF58476D1CE4E5B9 & 0xFFFFFFFFFFFFFFFF
        h = (h ^ (h >> 27)) * 0x94D049BB133111EB & 0xFFFFFFFFFFFFFFFF
        h ^= h >> 31
    return h & 0x7FFFFFFFFFFFFFFF


def kv_block(cfg: WorkloadConfig, layer: int, seq_index: int, n_tokens: int, kind: str,
             device="cpu"):
    """K (kind='k') or V (kind='v') of the cached prefix of one sequence in
    one layer pool: bf16 [n_tokens, H_kv, d], logical token order."""
    code = {"k": 1, "v": 2}[kind]
    return _draw((n_tokens, cfg.num_kv_heads, cfg.head_dim), cfg.kv_scale,
                 _mix(cfg.seed, 11, layer, seq_index, code), device)


def packed_prefix(cfg: WorkloadConfig, layers, lens, device="cpu"):
    """The cached prefixes of a batch packed for one varlen bulk write:
    (k, v, cu_seqlens) with k, v bf16 [len(layers)][sum(lens)][H_kv][d] whose
    rows cu_seqlens[b] .. cu_seqlens[b+1]-1 in slab i are kv_block(cfg,
    layers[i], b, lens[b]); sequences in batch order."""
    import torch
    cu = [0]
    for n in lens:
        cu.append(cu[-1] + int(n))
    shape = (len(layers), cu[-1], cfg.num_kv_heads, cfg.head_dim)
    k = torch.empty(shape, dtype=torch.bfloat16, device=device)
    v = torch.empty(shape, dtype=torch.bfloat16, device=device)
    for i, layer in enumerate(layers):
        for b, n in enumerate(lens):
            if int(n):
                k[i, cu[b]:cu[b + 1]] = kv_block(cfg, layer, b, int(n), "k", device)
                v[i, cu[b]:cu[b + 1]] = kv_block(cfg, layer, b, int(n), "v", device)
    return k, v, cu


def step_inputs(cfg: WorkloadConfig, step: int, layer: int, device="cpu"):
    """(q [B, H_q, d], k_new [B, H_kv, d], v_new [B, H_kv, d]) bf16 for one
    decode step of one logical layer."""
    B, Hq, Hkv, d = cfg.batch, cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim
    q = _draw((B, Hq, d), cfg.q_scale, _mix(cfg.seed, 21, step, layer), device)
    k = _draw((B, Hkv, d), cfg.kv_scale, _mix(cfg.seed, 22, step, layer), device)
    v = _draw((B, Hkv, d), cfg.kv_scale, _mix(cfg.seed, 23, step, layer), device)
    return q, k, v


def algorithmic_bytes_per_layer(cfg: WorkloadConfig, attended_lens) -> int:
    """Bytes one layer of a decode step must move: K and V of every attended
    token, Q read, O written, and the appended K/V written (bf16)."""
    Hq, Hkv, d = cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim
    n_tok = int(sum(int(x) for x in attended_lens))
    B = len(attended_lens)
    return n_tok * 2 * Hkv * d * 2 + B * Hq * d * 2 * 2 + B * 2 * Hkv * d * 2
