"""Packed varlen bulk K/V write (kv_write_varlen) against the oracle's page
scatter: every byte of every layer pool after the call equals the oracle
applied to the pool before it (so nothing outside the written positions
moves), for partial pages at both ends of a block, several blocks per
sequence in any packed order, empty blocks, and batches of more than 512
blocks (several launches).  At the LLaVA-1.5-7B-shaped handoff size (64
sequences, 32 layers) the oracle's page gather returns the packed input."""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_12707_gb300 import kvdecode as kd
from paper_2603_12707_gb300 import workloads as wl
from paper_2603_12707_gb300.harness import DecodeSession

from _gpu_common import _CAI, assert_close, bf16_to_f64, u16

pytestmark = pytest.mark.gpu


def _pool(h, layer, num_pages, Hkv, d):
    kp, vp = kd.kv_cache_pool(h, layer)
    shape = (num_pages, Hkv, 16, d)
    k = torch.as_tensor(_CAI(kp, shape), device="cuda")
    v = torch.as_tensor(_CAI(vp, shape), device="cuda")
    torch.cuda.synchronize()
    return k, v


def _cache(L, Hq, Hkv, d, lens, seed, slack=3):
    pages = sum((n + 15) // 16 for n in lens) + slack
    max_pages = max(1, max((n + 15) // 16 for n in lens))
    h = kd.kv_cache_create(kd.make_config(L, Hq, Hkv, d, pages, len(lens), max_pages))
    kd.kv_cache_set_page_order(h, np.random.default_rng(seed).permutation(pages))
    seqs = [kd.kv_seq_create(h) for _ in lens]
    for s, n in zip(seqs, lens):
        kd.kv_seq_reserve(h, s, n)
    # known junk everywhere, so a stray write shows
    for l in range(L):
        for t in _pool(h, l, pages, Hkv, d):
            t.copy_(torch.randint(-32768, 32767, t.shape, dtype=torch.int16, device="cuda",
                                  generator=torch.Generator("cuda").manual_seed(seed + l)))
    torch.cuda.synchronize()
    return h, seqs, pages


def _check(h, seqs, pages, L, Hkv, d, layer_first, blocks, k, v, before):
    """blocks: (seq index, first_pos, packed row, n) per block."""
    for l in range(L):
        got_k, got_v = (u16(t) for t in _pool(h, l, pages, Hkv, d))
        exp_k, exp_v = before[l][0].copy(), before[l][1].copy()
        if layer_first <= l < layer_first + k.shape[0]:
            src_k, src_v = u16(k[l - layer_first]), u16(v[l - layer_first])
            for si, first, row, n in blocks:
                pt = np.asarray(kd.kv_seq_info(h, seqs[si])[1], dtype=np.int32)
                oracle.kv_scatter(exp_k, pt, first, src_k[row:row + n], 16)
                oracle.kv_scatter(exp_v, pt, first, src_v[row:row + n], 16)
        assert np.array_equal(got_k, exp_k), l
        assert np.array_equal(got_v, exp_v), l


def _run(Hq, Hkv, d, lens, split, seed, L=3, layer_first=1, n_layers=2):
    """split: per sequence, the cut points of its prefix into blocks."""
    h, seqs, pages = _cache(L, Hq, Hkv, d, lens, seed)
    blocks = []
    for si, n in enumerate(lens):
        cuts = [0] + list(split.get(si, [])) + [n]
        for a, b in zip(cuts[:-1], cuts[1:]):
            blocks.append((si, a, b - a))
    order = np.random.default_rng(seed + 1).permutation(len(blocks))
    blocks = [blocks[i] for i in order]
    cu = [0]
    for _, _, n in blocks:
        cu.append(cu[-1] + n)
    cfg = wl.custom("varlen", n_layers, Hq, Hkv, d, 1, lens=[1], seed=seed)
    k = torch.empty((n_layers, cu[-1], Hkv, d), dtype=torch.bfloat16, device="cuda")
    v = torch.empty_like(k)
    for i, (_, _, n) in enumerate(blocks):
        if n:
            for l in range(n_layers):
                k[l, cu[i]:cu[i + 1]] = wl.kv_block(cfg, l, i, n, "k", "cuda")
                v[l, cu[i]:cu[i + 1]] = wl.kv_block(cfg, l, i, n, "v", "cuda")
    before = [tuple(u16(t) for t in _pool(h, l, pages, Hkv, d)) for l in range(L)]
    n0 = kd.kv_cache_query(h).kernel_launches
    kd.kv_write_varlen(h, layer_first, n_layers, [seqs[si] for si, _, _ in blocks], cu, k, v,
                       first_pos=[a for _, a, _ in blocks])
    torch.cuda.synchronize()
    st = kd.kv_cache_query(h)
    assert st.device_error == 0
    nonempty = sum(1 for _, _, n in blocks if n)
    assert st.kernel_launches - n0 == (nonempty + 511) // 512
    _check(h, seqs, pages, L, Hkv, d, layer_first,
           [(si, a, cu[i], n) for i, (si, a, n) in enumerate(blocks)], k, v, before)
    kd.kv_cache_destroy(h)


@pytest.mark.parametrize("Hq,Hkv,d", [(8, 8, 64), (28, 4, 128), (32, 32, 128)])
def test_varlen_write_matches_oracle_scatter(kvlib, Hq, Hkv, d):
    lens = [1, 15, 16, 17, 100, 33, 47]
    # several blocks per sequence: mid-page cuts, a page-aligned cut, an empty block
    split = {3: [5], 4: [37, 48, 48], 6: [20]}
    _run(Hq, Hkv, d, lens, split, seed=7 + d + Hkv)


def test_varlen_write_many_blocks_span_launches(kvlib):
    # 700 one-token blocks of one sequence plus three whole prefixes: 703 blocks, two launches
    lens = [700, 31, 64, 5]
    _run(28, 4, 128, lens, {0: list(range(1, 700))}, seed=91, L=2, layer_first=0, n_layers=2)


def test_varlen_write_llava_handoff(kvlib):
    """The whole LLaVA-shaped batch's prefixes (64 sequences, 576 vision
    tokens + prompt + generated) into all 32 layer pools in one call; layers 0
    and 31 read back through the oracle's page gather."""
    cfg = wl.CONFIGS["llava"]
    sess = DecodeSession(cfg, extra_tokens=1)
    lens = [int(n) for n in sess.lens0]
    k, v, cu = wl.packed_prefix(cfg, range(cfg.num_layers), lens, "cuda")
    kd.kv_write_varlen(sess.h, 0, cfg.num_layers, sess.seq_ids, cu, k, v)
    torch.cuda.synchronize()
    assert sess.query().device_error == 0
    for l in (0, cfg.num_layers - 1):
        pk, pv = (u16(t) for t in _pool(sess.h, l, sess.num_pages, cfg.num_kv_heads, cfg.head_dim))
        src_k, src_v = u16(k[l]), u16(v[l])
        for b, s in enumerate(sess.seq_ids):
            pt = np.asarray(kd.kv_seq_info(sess.h, s)[1], dtype=np.int32)
            assert np.array_equal(oracle.kv_gather(pk, pt, 0, lens[b]), src_k[cu[b]:cu[b + 1]]), (l, b)
            assert np.array_equal(oracle.kv_gather(pv, pt, 0, lens[b]), src_v[cu[b]:cu[b + 1]]), (l, b)
    sess.close()


def test_decode_after_varlen_prefix_matches_oracle(kvlib):
    """The prefixes of a ragged GQA batch written by one kv_write_varlen call
    (all layers), then three fused decode steps: every output matches the
    oracle over the written prefix plus the appended tokens."""
    cfg = wl.custom("varlen_decode", 3, 28, 4, 128, 5, lens=[1, 16, 17, 300, 1000], seed=77,
                    page_order="shuffled")
    sess = DecodeSession(cfg, extra_tokens=4)
    lens = [int(n) for n in sess.lens0]
    k, v, cu = wl.packed_prefix(cfg, range(cfg.num_layers), lens, "cuda")
    kd.kv_write_varlen(sess.h, 0, cfg.num_layers, sess.seq_ids, cu, k, v)
    hk = {(l, b): list(u16(k[l, cu[b]:cu[b + 1]])) for l in range(cfg.num_layers) for b in range(cfg.batch)}
    hv = {(l, b): list(u16(v[l, cu[b]:cu[b + 1]])) for l in range(cfg.num_layers) for b in range(cfg.batch)}
    for step in range(3):
        sess.begin_step()
        for l in range(cfg.num_layers):
            q, kn, vn = wl.step_inputs(cfg, step, l, "cuda")
            out = torch.empty_like(q)
            sess.append_attend(l, q, kn, vn, out)
            torch.cuda.synchronize()
            for b in range(cfg.batch):
                hk[(l, b)].append(u16(kn)[b])
                hv[(l, b)].append(u16(vn)[b])
            kk = np.concatenate([np.stack(hk[(l, b)]) for b in range(cfg.batch)])
            vv = np.concatenate([np.stack(hv[(l, b)]) for b in range(cfg.batch)])
            ref = oracle.decode_attention(u16(q), [len(hk[(l, b)]) for b in range(cfg.batch)], kk, vv)
            vmax = np.array([np.abs(oracle.bf16_to_f64(np.stack(hv[(l, b)]))).max() for b in range(cfg.batch)])
            assert_close(bf16_to_f64(out), ref, vmax, gqa=True, what=(step, l))
    assert sess.query().device_error == 0
    sess.close()
