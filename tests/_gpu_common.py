"""Shared pieces of the GPU parity tests: a decode session that also keeps the
host copy of everything the cache should hold, so the oracle can be fed the
same logical-order K/V."""
import numpy as np
import torch

import oracle
from paper_2603_12707_gb300 import kvdecode as kd
from paper_2603_12707_gb300 import workloads as wl
from paper_2603_12707_gb300.harness import DecodeSession


def u16(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


class _CAI:
    """Expose a raw device allocation to torch (int16 view) for read-back."""

    def __init__(self, ptr, shape):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": "<i2", "data": (int(ptr), False),
                                         "version": 3, "strides": None}


def device_pool(sess: DecodeSession, layer: int):
    """Raw K and V pools of one layer as uint16 [num_pages, H_kv, P, d] host arrays."""
    kp, vp = kd.kv_cache_pool(sess.h, layer)
    c = sess.cfg
    shape = (sess.num_pages, c.num_kv_heads, c.page_size, c.head_dim)
    k = torch.as_tensor(_CAI(kp, shape), device="cuda")
    v = torch.as_tensor(_CAI(vp, shape), device="cuda")
    torch.cuda.synchronize()
    return u16(k), u16(v)


class Tracked:
    """A DecodeSession plus host copies of each layer pool's logical content."""

    def __init__(self, cfg, extra_tokens=8, lens=None, split_pages=0, layers_filled=None, keep_host=True,
                 keep_rows=None, stream=None):
        self.cfg = cfg
        self.sess = DecodeSession(cfg, extra_tokens=extra_tokens, lens=lens, split_pages=split_pages, stream=stream)
        self.keep_host = keep_host
        self.keep_rows = list(range(cfg.batch)) if keep_rows is None else list(keep_rows)
        self.layers_filled = list(range(cfg.phys_layers)) if layers_filled is None else list(layers_filled)
        self.sess.fill_prefix(self.layers_filled)
        # host logical content per (phys layer, batch row): list of token rows [H_kv, d]
        self.k = {}
        self.v = {}
        if keep_host:
            for l in self.layers_filled:
                for b in self.keep_rows:
                    n = int(self.sess.lens0[b])
                    self.k[(l, b)] = list(u16(wl.kv_block(cfg, l, b, n, "k", "cuda"))) if n else []
                    self.v[(l, b)] = list(u16(wl.kv_block(cfg, l, b, n, "v", "cuda"))) if n else []
        self.step = -1

    def begin_step(self):
        self.sess.begin_step()
        self.step += 1

    def run_layer(self, layer, scale=0.0, fused=False):
        """Append + attend one logical layer (two launches, or the fused one);
        returns (out bf16 tensor, q, k_new, v_new)."""
        cfg = self.cfg
        q, kn, vn = wl.step_inputs(cfg, self.step, layer, "cuda")
        out = torch.empty_like(q)
        if fused:
            self.sess.append_attend(layer, q, kn, vn, out, scale)
        else:
            self.sess.append(layer, kn, vn)
            self.sess.attend(layer, q, out, scale)
        if self.keep_host:
            p = self.sess.phys(layer)
            kh, vh = u16(kn), u16(vn)
            for b in self.keep_rows:
                pos = int(self.sess.lens[b]) - 1
                for store, val in ((self.k, kh[b]), (self.v, vh[b])):
                    rows = store[(p, b)]
                    if pos == len(rows):
                        rows.append(val)
                    else:
                        rows[pos] = val
        return out, q, kn, vn

    def oracle(self, layer, q, rows=None, scale=None):
        """float64 oracle output for the given batch rows of one layer."""
        p = self.sess.phys(layer)
        rows = list(range(self.cfg.batch)) if rows is None else list(rows)
        lens = [len(self.k[(p, b)]) for b in rows]
        k = np.concatenate([np.stack(self.k[(p, b)]) for b in rows])
        v = np.concatenate([np.stack(self.v[(p, b)]) for b in rows])
        qh = u16(q)[rows]
        ref = oracle.decode_attention(qh, lens, k, v, scale=scale)
        vmax = np.array([np.abs(oracle.bf16_to_f64(np.stack(self.v[(p, b)]))).max() for b in rows])
        return ref, vmax

    def close(self):
        st = self.sess.query()
        assert st.device_error == 0
        self.sess.close()


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().double().numpy()


def assert_close(got, ref, vmax, gqa: bool, what=""):
    """Spec bound (max |err| <= 2e-2, mean |err| <= 2e-3) and the bound
    derived from the arithmetic: bf16 rounding of the output (2^-8 relative),
    bf16 rounding of the softmax weights fed to the P.V MMA (GQA only: each
    weight p_t moves by at most 2^-8 p_t, bf16's unit roundoff, so the
    normalised output moves by at most sum_t 2^-8 p_t |v_t| / sum_t p_t <=
    2^-8 * max|v|) and fp32 accumulation (1e-5 * max|v|)."""
    err = np.abs(got - ref)
    assert err.max() <= 2e-2, (what, err.max())
    assert err.mean() <= 2e-3, (what, err.mean())
    w = (2.0 ** -8 if gqa else 0.0) + 1e-5
    bound = 2.0 ** -8 * np.abs(ref) + w * vmax[:, None, None]
    bad = err > bound
    assert not bad.any(), (what, int(bad.sum()), float((err - bound).max()), np.argwhere(bad)[:5].tolist())


# NaN, -NaN, +Inf and -Inf as bf16 bit patterns (int16 view)
POISON = (0x7FC0, 0xFFC0 - 0x10000, 0x7F80, 0xFF80 - 0x10000)


def poison_unused_slots(sess: DecodeSession):
    """Fill every pool slot that no sequence holds (the free pages, and the
    slots past each sequence's length on its last page) with NaN / Inf bit
    patterns in every layer's K and V pools, so a result that let one of them
    in shows it.  Returns the number of slots poisoned per pool."""
    c = sess.cfg
    P = c.page_size
    used = np.zeros((sess.num_pages, P), bool)
    for seq in sess.seq_ids:
        n, pages = kd.kv_seq_info(sess.h, seq)
        for i, pg in enumerate(pages):
            k = min(P, n - i * P)
            if k > 0:
                used[pg, :k] = True
    idx = np.arange(sess.num_pages)[:, None] + np.arange(P)[None, :]
    patt = np.array(POISON, np.int16)[idx % len(POISON)]
    mask = torch.from_numpy(~used).cuda()[:, None, :, None]
    fill = torch.from_numpy(patt).cuda()[:, None, :, None]
    shape = (sess.num_pages, c.num_kv_heads, P, c.head_dim)
    for layer in range(c.phys_layers):
        for ptr in kd.kv_cache_pool(sess.h, layer):
            pool = torch.as_tensor(_CAI(ptr, shape), device="cuda")
            pool.copy_(torch.where(mask, fill, pool))
    torch.cuda.synchronize()
    return int((~used).sum())
