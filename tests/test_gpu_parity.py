"""GPU parity of the CUDA path against the float64 oracle, through the C ABI.

* kv_append and the prefix write: bit-exact pool contents and page tables.
* decode_attention: every output element against the oracle, on small
  configs that span several pages, splits and a ragged tail, on the edge
  cases (a fresh sequence attending one token, page-boundary lengths, one
  page per split, unsplit rows), and on sampled rows of the five workload
  shapes at full size in the launch configuration the bench uses.
"""
import numpy as np
import pytest
import torch

import oracle
from oracle import PagePoolModel
from paper_2603_12707_gb300 import kvdecode as kd
from paper_2603_12707_gb300 import workloads as wl

from _gpu_common import Tracked, assert_close, bf16_to_f64, device_pool, u16

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True, scope="module")
def _lib(kvlib):
    assert torch.cuda.is_available()
    yield


def _model_for(sess):
    c = sess.cfg
    m = PagePoolModel(sess.num_pages, c.page_size, c.batch, sess.max_pages)
    order = wl.page_order(c, sess.num_pages)
    if order is not None:
        m.set_page_order(order)
    for _ in range(c.batch):
        m.seq_create()
    for i, n in wl.reserve_schedule(c, sess.lens0):
        m.seq_reserve(i, n)
    return m


# ---------------------------------------------------------------- kv_append
@pytest.mark.parametrize("cfg", [
    wl.CONFIGS["tiny"],
    wl.custom("gqa128", 2, 14, 2, 128, 5, lens=[0, 15, 16, 17, 40], page_order="interleaved"),
    wl.custom("mha64", 1, 4, 4, 64, 3, lens=[31, 32, 1], page_order="shuffled", seed=9),
])
def test_prefix_write_and_append_are_bit_exact(cfg):
    t = Tracked(cfg, extra_tokens=40)
    sess = t.sess
    model = _model_for(sess)
    for step in range(3):
        t.begin_step()
        model.begin_step(list(range(cfg.batch)))
        for layer in range(cfg.num_layers):
            t.run_layer(layer)
    torch.cuda.synchronize()
    # page tables: library == oracle allocator model, entry for entry
    for b, seq in enumerate(sess.seq_ids):
        ln, pages = kd.kv_seq_info(sess.h, seq)
        assert ln == model.lens[b] and pages == model.pages[b]
    # pools: the oracle scatters the same logical rows through the model's tables
    for l in range(cfg.phys_layers):
        shape = (sess.num_pages, cfg.num_kv_heads, cfg.page_size, cfg.head_dim)
        ek, ev = np.zeros(shape, np.uint16), np.zeros(shape, np.uint16)
        for b in range(cfg.batch):
            row = np.array(model.pages[b], np.int32)
            if len(t.k[(l, b)]):
                oracle.kv_scatter(ek, row, 0, np.stack(t.k[(l, b)]), cfg.page_size)
                oracle.kv_scatter(ev, row, 0, np.stack(t.v[(l, b)]), cfg.page_size)
        gk, gv = device_pool(sess, l)
        assert np.array_equal(gk, ek) and np.array_equal(gv, ev)
        # read-back through the ABI returns the logical rows
        for b, seq in enumerate(sess.seq_ids):
            n = int(sess.lens[b])
            ko = torch.empty((n, cfg.num_kv_heads, cfg.head_dim), dtype=torch.bfloat16, device="cuda")
            vo = torch.empty_like(ko)
            kd.kv_read_tokens(sess.h, l, seq, 0, n, ko, vo)
            assert np.array_equal(u16(ko), np.stack(t.k[(l, b)]))
            assert np.array_equal(u16(vo), np.stack(t.v[(l, b)]))
    t.close()


# ---------------------------------------------------------- decode: small
SMALL = [
    # name, Hq, Hkv, d, lens (cached before the first step)
    ("mha64", 8, 8, 64, [0, 1, 15, 16, 17, 95, 130]),
    ("mha128", 4, 4, 128, [0, 15, 16, 31, 200, 513]),
    ("gqa7_128", 28, 4, 128, [0, 1, 16, 47, 300]),
    ("gqa7_64", 14, 2, 64, [3, 16, 33, 250]),
    ("gqa8_64", 8, 1, 64, [5, 64, 129]),
    ("gqa2_128", 4, 2, 128, [17, 100, 1000]),
    # the other group sizes the MMA tile pads to 8 query heads
    ("gqa3_64", 6, 2, 64, [2, 31, 160]),
    ("gqa4_128", 16, 4, 128, [16, 65, 333]),
    ("gqa5_128", 10, 2, 128, [1, 48, 511]),
    ("gqa6_64", 12, 2, 64, [9, 80, 257]),
    ("gqa8_128", 8, 1, 128, [31, 250, 1100]),
    # the head shapes of the larger backends in the paper's footprint table (Table 3):
    # LLaVA-13B (MHA 40/40) and LLaVA-34B (GQA 56 query heads over 8 KV heads), d 128
    ("llava13b", 40, 40, 128, [7, 16, 577, 1200]),
    ("llava34b", 56, 8, 128, [1, 32, 640, 2000]),
    # rows longer than a 32-page id window, and longer than the item cap at small splits
    ("mha64_long", 8, 8, 64, [3000, 40]),
    ("gqa7_long", 28, 4, 128, [4000, 5]),
    ("gqa7_64_long", 14, 2, 64, [2600, 33, 700]),   # d 64: a 6-stage ring across id windows
]


@pytest.mark.parametrize("max_items", [2, 3, 7, 12, 20, 32, 33, 48, 64])
@pytest.mark.parametrize("Hq,Hkv,d", [(8, 8, 128), (28, 4, 128), (14, 2, 64)])
def test_merge_batch_variants(Hq, Hkv, d, max_items):
    """The merge pass is compiled for 4, 8, 16 or 32 items in flight and the
    launch picks the smallest that covers the step's longest row: one-page
    items and a longest row of max_items pages exercise each variant, with
    shorter rows (one item, several items) beside it.  These batches have
    few rows, so rows may hold up to 64 items: 33, 48 and 64 take the
    four-warp variant (16 items per warp, combined in shared memory; at 33 a
    warp with one item and an idle warp)."""
    lens = [16 * max_items - 1, 40, 5, 16 * max(1, max_items // 2)]
    cfg = wl.custom(f"merge{max_items}", 1, Hq, Hkv, d, len(lens), lens=lens, seed=400 + max_items,
                    page_order="shuffled")
    t = Tracked(cfg, extra_tokens=4, split_pages=1)
    for _ in range(2):
        t.begin_step()
        for fused in (False, True):
            out, q, _, _ = t.run_layer(0, fused=fused)
            torch.cuda.synchronize()
            ref, vmax = t.oracle(0, q)
            assert_close(bf16_to_f64(out), ref, vmax, gqa=Hq > Hkv, what=(max_items, fused))
            if not fused:
                t.begin_step()
    t.close()


@pytest.mark.parametrize("split", [0, 1, 3, 64, 1024])
@pytest.mark.parametrize("name,Hq,Hkv,d,lens", SMALL)
def test_decode_matches_oracle_small(name, Hq, Hkv, d, lens, split):
    cfg = wl.custom(name, 2, Hq, Hkv, d, len(lens), lens=lens, seed=31 + Hq + d, page_order="shuffled")
    t = Tracked(cfg, extra_tokens=20, split_pages=split)
    for step in range(3):
        t.begin_step()
        for layer in range(cfg.num_layers):
            out, q, _, _ = t.run_layer(layer)
            torch.cuda.synchronize()
            ref, vmax = t.oracle(layer, q)
            assert_close(bf16_to_f64(out), ref, vmax, gqa=Hq > Hkv, what=(name, split, step, layer))
    t.close()


@pytest.mark.parametrize("Hq,Hkv,d", [(8, 8, 128), (28, 4, 128), (6, 2, 64)])
def test_rows_filled_to_the_last_page_slot(Hq, Hkv, d):
    """Page-table rows of exactly 4 pages: the third step's row 0 attends all
    64 positions its row can hold (the last slot of the last page)."""
    cfg = wl.custom("fullrow", 1, Hq, Hkv, d, 3, lens=[61, 13, 47], seed=61 + d)
    t = Tracked(cfg, extra_tokens=3, split_pages=1)
    assert t.sess.max_pages == 4
    for step in range(3):
        t.begin_step()
        out, q, _, _ = t.run_layer(0, fused=(step % 2 == 1))
        torch.cuda.synchronize()
        ref, vmax = t.oracle(0, q)
        assert_close(bf16_to_f64(out), ref, vmax, gqa=Hq > Hkv, what=(step,))
    assert kd.kv_seq_info(t.sess.h, t.sess.seq_ids[0])[0] == 64
    t.close()


@pytest.mark.parametrize("scale", [0.37, 1e-4])
@pytest.mark.parametrize("Hq,Hkv", [(14, 2), (8, 8)])
def test_custom_softmax_scale(Hq, Hkv, scale):
    """A caller's scale; at 1e-4 every weight is nearly equal and the output is
    close to the mean of V (the degenerate uniform softmax)."""
    cfg = wl.custom("scale", 1, Hq, Hkv, 128, 3, lens=[10, 40, 90], seed=5)
    t = Tracked(cfg, split_pages=2)
    t.begin_step()
    out, q, _, _ = t.run_layer(0, scale=scale)
    torch.cuda.synchronize()
    ref, vmax = t.oracle(0, q, scale=scale)
    assert_close(bf16_to_f64(out), ref, vmax, gqa=Hq > Hkv)
    t.close()


@pytest.mark.parametrize("fused", [False, True])
@pytest.mark.parametrize("split", [0, 1, 3])
@pytest.mark.parametrize("Hq,Hkv,d", [(28, 4, 128), (8, 8, 64), (6, 2, 64)])
def test_wide_score_range_moves_the_running_max(Hq, Hkv, d, split, fused):
    """softmax_scale 3 makes the scores N(0, (3 sqrt(d))^2): the running max of
    a head keeps jumping by far more than 2^8 across pages and items, so every
    rescale path of the split pass and the merge runs."""
    cfg = wl.custom("wide", 1, Hq, Hkv, d, 3, lens=[300, 700, 47], seed=41 + d, page_order="shuffled")
    t = Tracked(cfg, split_pages=split)
    t.begin_step()
    out, q, _, _ = t.run_layer(0, scale=3.0, fused=fused)
    torch.cuda.synchronize()
    ref, vmax = t.oracle(0, q, scale=3.0)
    assert_close(bf16_to_f64(out), ref, vmax, gqa=Hq > Hkv, what=(Hq, Hkv, d, split, fused))
    t.close()


def test_single_token_context_returns_appended_v():
    """A sequence with nothing cached attends only its new token: out == v_new
    exactly (weights are exactly 1, and bf16 -> fp32 -> bf16 is lossless)."""
    for Hq, Hkv, d in ((8, 8, 64), (28, 4, 128)):
        cfg = wl.custom("one", 1, Hq, Hkv, d, 3, lens=[0, 0, 0], seed=3)
        t = Tracked(cfg)
        t.begin_step()
        out, q, kn, vn = t.run_layer(0)
        torch.cuda.synchronize()
        G = Hq // Hkv
        expect = vn.repeat_interleave(G, dim=1)
        assert torch.equal(out, expect)
        t.close()


def test_page_order_does_not_change_results():
    """Same logical content in different physical pages: bit-identical output."""
    outs = []
    for order in ("sequential", "shuffled", "interleaved"):
        cfg = wl.custom("perm", 1, 28, 4, 128, 4, lens=[100, 37, 260, 16], seed=77, page_order=order)
        t = Tracked(cfg, keep_host=False)
        t.begin_step()
        out, _, _, _ = t.run_layer(0)
        torch.cuda.synchronize()
        outs.append(out.clone())
        t.close()
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


def test_split_size_changes_only_rounding():
    res = {}
    for split in (1, 4, 64):
        cfg = wl.custom("split", 1, 8, 8, 128, 3, lens=[700, 33, 1023], seed=13)
        t = Tracked(cfg, split_pages=split, keep_host=False)
        t.begin_step()
        out, _, _, _ = t.run_layer(0)
        torch.cuda.synchronize()
        res[split] = bf16_to_f64(out)
        t.close()
    for s in (1, 4):
        d = np.abs(res[s] - res[64])
        assert d.max() <= 2.0 ** -7 * np.abs(res[64]).max()


def test_step_and_attention_errors_do_not_launch():
    cfg = wl.custom("err", 1, 8, 8, 64, 2, lens=[5, 9], seed=1)
    t = Tracked(cfg, keep_host=False)
    q = torch.zeros((2, 8, 64), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(q)
    with pytest.raises(kd.KVDecodeError):           # no step yet
        kd.decode_attention(t.sess.h, 0, 2, q, out)
    t.begin_step()
    with pytest.raises(kd.KVDecodeError):           # wrong batch
        kd.decode_attention(t.sess.h, 0, 1, q, out)
    with pytest.raises(kd.KVDecodeError):           # bad layer
        kd.kv_append(t.sess.h, 3, 2, q, q)
    with pytest.raises(kd.KVDecodeError):           # misaligned pointer
        kd.decode_attention(t.sess.h, 0, 2, q.data_ptr() + 2, out)
    t.close()


# ------------------------------------------------------ fused append + attend
@pytest.mark.parametrize("name,Hq,Hkv,d,lens", [
    ("mha128", 8, 8, 128, [0, 15, 16, 31, 200, 700]),
    ("gqa7_128", 28, 4, 128, [0, 1, 16, 47, 300, 2100]),
    ("mha64", 8, 8, 64, [3, 16, 129]),
    ("gqa7_64", 14, 2, 64, [15, 33, 250]),
])
@pytest.mark.parametrize("split", [0, 1, 1024])
def test_fused_append_attend_equals_append_then_attend(name, Hq, Hkv, d, lens, split):
    """decode_attention_append: bit-identical output and cache contents to
    kv_append + decode_attention, and the oracle's result, over several
    steps (pages filling up and new pages taken)."""
    outs = {}
    pools = {}
    for fused in (False, True):
        cfg = wl.custom(name, 3, Hq, Hkv, d, len(lens), lens=lens, seed=41 + d, page_order="shuffled")
        t = Tracked(cfg, extra_tokens=24, split_pages=split, keep_host=fused)
        res = []
        for step in range(4):
            t.begin_step()
            for layer in range(cfg.num_layers):
                out, q, _, _ = t.run_layer(layer, fused=fused)
                res.append(out.clone())
                if fused and step in (0, 3):
                    torch.cuda.synchronize()
                    ref, vmax = t.oracle(layer, q)
                    assert_close(bf16_to_f64(out), ref, vmax, gqa=Hq > Hkv, what=(name, split, step, layer))
        torch.cuda.synchronize()
        outs[fused] = res
        pools[fused] = [device_pool(t.sess, l) for l in range(cfg.phys_layers)]
        t.close()
    for a, b in zip(outs[False], outs[True]):
        assert torch.equal(a, b)
    for (ka, va), (kb, vb) in zip(pools[False], pools[True]):
        assert np.array_equal(ka, kb) and np.array_equal(va, vb)


def test_fused_layers_back_to_back_on_one_stream():
    """Consecutive fused launches overlap (each may start while the previous
    drains): a whole multi-layer step on one side stream matches the oracle."""
    cfg = wl.custom("pdl", 6, 28, 4, 128, 6, lens=[900, 33, 2500, 16, 400, 1200], seed=99, page_order="shuffled")
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        t = Tracked(cfg, extra_tokens=8, stream=stream)
        for step in range(2):
            t.begin_step()
            got = []
            for layer in range(cfg.num_layers):
                out, q, _, _ = t.run_layer(layer, fused=True)
                got.append((layer, out, q))
            stream.synchronize()
            for layer, out, q in got:
                ref, vmax = t.oracle(layer, q)
                assert_close(bf16_to_f64(out), ref, vmax, gqa=True, what=(step, layer))
        t.close()


# ------------------------------------------------------- decode: full size
FULL = [
    # config, logical layers checked, sampled batch rows
    ("tiny", [0], None),
    ("llava", [0, 17, 31], [0, 1, 2, 63]),
    ("qwen", [0, 27], [0, 5, 31]),
    ("long", [0, 27], [0, 7]),
    ("ragged", [0, 9, 31], [0, 100, 255]),
]


@pytest.mark.parametrize("name,layers,rows", FULL)
def test_decode_matches_oracle_full_size(name, layers, rows):
    cfg = wl.CONFIGS[name]
    phys = sorted({l % cfg.phys_layers for l in layers})
    t = Tracked(cfg, extra_tokens=4, layers_filled=phys, keep_rows=rows)
    t.begin_step()
    for i, layer in enumerate(layers):
        out, q, _, _ = t.run_layer(layer, fused=(i % 2 == 1))
        torch.cuda.synchronize()
        r = list(range(cfg.batch)) if rows is None else rows
        ref, vmax = t.oracle(layer, q, rows=r)
        assert_close(bf16_to_f64(out)[r], ref, vmax, gqa=cfg.group > 1, what=(name, layer))
    t.close()


# -------------------------------- full size, in the bench's launch configuration
FULL_GRAPH = [
    # config, logical layers checked (distinct pools; for the ragged config the
    # last logical layer of each checked pool), sampled batch rows
    ("llava", [0, 31], [0, 1, 63]),
    ("qwen", [0, 27], [0, 5, 31]),
    ("long", [0, 27], [0, 7]),
    ("ragged", [24, 31], [0, 100, 255]),
]


@pytest.mark.parametrize("name,layers,rows", FULL_GRAPH)
def test_graph_replayed_steps_match_oracle_full_size(name, layers, rows):
    """Device-side steps and all L fused layers captured into CUDA graphs and
    replayed, as bench.py times them; after one eager and three replayed
    steps every checked layer's output matches the oracle over the prefix
    plus the four appended tokens."""
    cfg = wl.CONFIGS[name]
    L, B = cfg.num_layers, cfg.batch
    phys = sorted({l % cfg.phys_layers for l in layers})
    assert len(phys) == len(layers)
    t = Tracked(cfg, extra_tokens=8, layers_filled=phys, keep_rows=rows)
    sess = t.sess
    s = torch.cuda.Stream()
    ins = [wl.step_inputs(cfg, 0, l, "cuda") for l in range(L)]
    outs = [torch.empty_like(i[0]) for i in ins]
    ids = torch.tensor(sess.seq_ids, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    kd.kv_cache_device_steps(sess.h, B, True, s)

    def all_layers():
        for l in range(L):
            kd.decode_attention_append(sess.h, sess.phys(l), B, ins[l][0], ins[l][1], ins[l][2], outs[l], 0.0, s)

    with torch.cuda.stream(s):
        kd.kv_begin_step_device(sess.h, B, ids, s)
        all_layers()
    s.synchronize()
    g_step, g_layers = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_step, stream=s):
        kd.kv_begin_step_device(sess.h, B, ids, s)
    with torch.cuda.graph(g_layers, stream=s):
        all_layers()
    with torch.cuda.stream(s):
        for _ in range(3):
            g_step.replay()
            g_layers.replay()
    s.synchronize()
    steps = 4
    kd.kv_cache_sync(sess.h)
    for b in rows:
        assert kd.kv_seq_info(sess.h, sess.seq_ids[b])[0] == int(sess.lens0[b]) + steps
    for l in layers:
        p = sess.phys(l)
        kh, vh = u16(ins[l][1]), u16(ins[l][2])
        for b in rows:
            t.k[(p, b)] += [kh[b]] * steps
            t.v[(p, b)] += [vh[b]] * steps
        ref, vmax = t.oracle(l, ins[l][0], rows=rows)
        assert_close(bf16_to_f64(outs[l])[rows], ref, vmax, gqa=cfg.group > 1, what=(name, l))
    t.close()
