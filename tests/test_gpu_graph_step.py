"""Device-side decode steps (kv_begin_step_device) and a whole decode step
captured once into a CUDA graph and replayed: same pages, same lengths and
bit-identical outputs as host-driven steps; exhaustion is reported."""
import numpy as np
import pytest
import torch

from oracle import PagePoolModel
from paper_2603_12707_gb300 import kvdecode as kd
from paper_2603_12707_gb300 import workloads as wl

from _gpu_common import Tracked, assert_close, bf16_to_f64

pytestmark = pytest.mark.gpu

SPLIT = 3   # same work-item size for both sides, so outputs are bit-identical


def _pair(cfg, extra=24):
    a = Tracked(cfg, extra_tokens=extra, split_pages=SPLIT, keep_host=True)
    b = Tracked(cfg, extra_tokens=extra, split_pages=SPLIT, keep_host=False)
    return a, b


@pytest.mark.parametrize("Hq,Hkv,d,lens", [
    (8, 8, 128, [0, 15, 16, 31, 200, 47]),
    (28, 4, 128, [1, 16, 300, 2100]),
])
def test_device_steps_match_host_steps(kvlib, Hq, Hkv, d, lens):
    cfg = wl.custom("devstep", 2, Hq, Hkv, d, len(lens), lens=lens, seed=5 + Hq, page_order="shuffled")
    a, b = _pair(cfg)
    kd.kv_cache_device_steps(b.sess.h, cfg.batch)
    ids = torch.tensor(b.sess.seq_ids, dtype=torch.int32, device="cuda")
    for step in range(20):
        a.begin_step()
        kd.kv_begin_step_device(b.sess.h, cfg.batch, ids)
        b.step += 1
        b.sess.lens += 1
        for layer in range(cfg.num_layers):
            oa, q, _, _ = a.run_layer(layer, fused=True)
            ob, _, _, _ = b.run_layer(layer, fused=(layer % 2 == 0))
            torch.cuda.synchronize()
            assert torch.equal(oa, ob), (step, layer)
            if step in (0, 19):
                ref, vmax = a.oracle(layer, q)
                assert_close(bf16_to_f64(ob), ref, vmax, gqa=Hq > Hkv)
    # the host view after a sync: same lengths and pages as host steps
    kd.kv_cache_sync(b.sess.h)
    for sa, sb in zip(a.sess.seq_ids, b.sess.seq_ids):
        assert kd.kv_seq_info(a.sess.h, sa) == kd.kv_seq_info(b.sess.h, sb)
    st_a, st_b = kd.kv_cache_query(a.sess.h), kd.kv_cache_query(b.sess.h)
    assert (st_a.pages_in_use, st_a.free_pages) == (st_b.pages_in_use, st_b.free_pages)
    # host calls keep working after device steps (allocator state came back)
    b.begin_step()
    a.begin_step()
    for sa, sb in zip(a.sess.seq_ids, b.sess.seq_ids):
        assert kd.kv_seq_info(a.sess.h, sa) == kd.kv_seq_info(b.sess.h, sb)
    a.close()
    b.close()


def test_captured_step_replays_like_host_steps(kvlib):
    cfg = wl.custom("graph", 4, 28, 4, 128, 5, lens=[100, 16, 999, 35, 512], seed=61, page_order="shuffled")
    a, b = _pair(cfg, extra=40)
    L = cfg.num_layers
    ins = [wl.step_inputs(cfg, 0, l, "cuda") for l in range(L)]
    outs = [torch.empty_like(i[0]) for i in ins]
    ids = torch.tensor(b.sess.seq_ids, dtype=torch.int32, device="cuda")
    kd.kv_cache_device_steps(b.sess.h, cfg.batch)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        # one eager step first so no lazy initialisation happens inside the capture
        kd.kv_begin_step_device(b.sess.h, cfg.batch, ids, s)
        for l in range(L):
            kd.decode_attention_append(b.sess.h, l, cfg.batch, ins[l][0], ins[l][1], ins[l][2], outs[l], 0.0, s)
    s.synchronize()
    a.sess.begin_step()
    for l in range(L):
        oa = torch.empty_like(outs[l])
        a.sess.append_attend(l, ins[l][0], ins[l][1], ins[l][2], oa)
        torch.cuda.synchronize()
        assert torch.equal(oa, outs[l])
    with torch.cuda.graph(g, stream=s):
        cs = torch.cuda.current_stream()
        kd.kv_begin_step_device(b.sess.h, cfg.batch, ids, cs)
        for l in range(L):
            kd.decode_attention_append(b.sess.h, l, cfg.batch, ins[l][0], ins[l][1], ins[l][2], outs[l], 0.0, cs)
    for rep in range(12):
        g.replay()
        a.sess.begin_step()
        refs = []
        for l in range(L):
            oa = torch.empty_like(outs[l])
            a.sess.append_attend(l, ins[l][0], ins[l][1], ins[l][2], oa)
            refs.append(oa)
        torch.cuda.synchronize()
        for l in range(L):
            assert torch.equal(refs[l], outs[l]), (rep, l)
    kd.kv_cache_sync(b.sess.h)
    for sa, sb in zip(a.sess.seq_ids, b.sess.seq_ids):
        assert kd.kv_seq_info(a.sess.h, sa) == kd.kv_seq_info(b.sess.h, sb)
    a.close()
    b.close()


def test_device_step_reports_an_exhausted_pool(kvlib):
    """5 pages, 3 sequences of 16 tokens (3 pages held): the next step needs a
    page for each; the first two rows (batch order) get them, the third is
    left at its length and the pool exhaustion is reported.  The fused layer
    launched after it appends the new token of the first two rows and leaves
    the third row's cache untouched (its last cached token is not
    overwritten)."""
    cfg = kd.make_config(1, 8, 8, 64, 5, 4, 8)
    h = kd.kv_cache_create(cfg)
    seqs = [kd.kv_seq_create(h) for _ in range(3)]
    gen = torch.Generator().manual_seed(3)
    cached = []
    for s_ in seqs:
        kd.kv_seq_reserve(h, s_, 16)
        k = torch.randn(16, 8, 64, generator=gen).to(torch.bfloat16).cuda()
        v = torch.randn(16, 8, 64, generator=gen).to(torch.bfloat16).cuda()
        kd.kv_write_tokens(h, 0, s_, 0, 16, k, v)
        cached.append((k, v))
    kd.kv_cache_device_steps(h, 3)
    ids = torch.tensor(seqs, dtype=torch.int32, device="cuda")
    kd.kv_begin_step_device(h, 3, ids)
    q = torch.randn(3, 8, 64, generator=gen).to(torch.bfloat16).cuda()
    kn = torch.randn(3, 8, 64, generator=gen).to(torch.bfloat16).cuda()
    vn = torch.randn(3, 8, 64, generator=gen).to(torch.bfloat16).cuda()
    out = torch.zeros(3, 8, 64, dtype=torch.bfloat16, device="cuda")
    kd.decode_attention_append(h, 0, 3, q, kn, vn, out)
    torch.cuda.synchronize()
    with pytest.raises(kd.KVDecodeError) as ei:
        kd.kv_cache_query(h)
    assert ei.value.code == kd.KVC_ERR_OOM
    st = kd.kv_cache_query(h, raise_on_device_error=False)
    assert st.device_error & kd.KVC_DEVERR_OOM
    assert st.free_pages == 0 and st.pages_in_use == 5
    assert [kd.kv_seq_info(h, s_)[0] for s_ in seqs] == [17, 17, 16]
    # the host allocator model agrees on which pages went where
    m = PagePoolModel(5, 16, 4, 8)
    for _ in range(3):
        m.seq_create()
    for i in range(3):
        m.seq_reserve(i, 16)
    m.seq_reserve(0, 1)
    m.seq_reserve(1, 1)
    for i, s_ in enumerate(seqs):
        assert kd.kv_seq_info(h, s_)[1] == m.pages[i]
    for i, s_ in enumerate(seqs):
        n = 17 if i < 2 else 16
        k = torch.empty(n, 8, 64, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        kd.kv_read_tokens(h, 0, s_, 0, n, k, v)
        torch.cuda.synchronize()
        assert torch.equal(k[:16], cached[i][0]) and torch.equal(v[:16], cached[i][1]), i
        if i < 2:
            assert torch.equal(k[16], kn[i]) and torch.equal(v[16], vn[i]), i
    kd.kv_cache_destroy(h)


def test_device_step_skips_an_unknown_sequence_id(kvlib):
    """A device-side sequence id outside the cache sets KVC_DEVERR_SEQ_RANGE;
    the other rows step and attend as usual (against the oracle)."""
    cfg = wl.custom("badid", 1, 8, 8, 64, 3, lens=[20, 33, 9], seed=23)
    t = Tracked(cfg, extra_tokens=4)
    kd.kv_cache_device_steps(t.sess.h, 3)
    s0, s1, s2 = t.sess.seq_ids
    ids = torch.tensor([s0, 77, s2], dtype=torch.int32, device="cuda")
    kd.kv_begin_step_device(t.sess.h, 3, ids)
    gen = torch.Generator().manual_seed(4)
    q3, kn3, vn3 = (torch.randn(3, 8, 64, generator=gen).to(torch.bfloat16).cuda() for _ in range(3))
    out3 = torch.zeros(3, 8, 64, dtype=torch.bfloat16, device="cuda")
    kd.decode_attention_append(t.sess.h, 0, 3, q3, kn3, vn3, out3)
    torch.cuda.synchronize()
    st = kd.kv_cache_query(t.sess.h, raise_on_device_error=False)
    assert st.device_error == kd.KVC_DEVERR_SEQ_RANGE
    assert [kd.kv_seq_info(t.sess.h, s_)[0] for s_ in (s0, s1, s2)] == [21, 33, 10]
    # launch rows 0 and 2 are sequences 0 and 2, each with its new token
    for b in (0, 2):
        for store, val in ((t.k, kn3[b]), (t.v, vn3[b])):
            store[(0, b)].append(val.view(torch.int16).cpu().numpy().view(np.uint16))
    ref, vmax = t.oracle(0, q3, rows=[0, 2])
    assert_close(bf16_to_f64(out3)[[0, 2]], ref, vmax, gqa=False)
    t.sess.close()


def test_device_steps_interleaved_with_host_lifecycle(kvlib):
    """Device-side steps mixed with host-side lifecycle calls (free a
    sequence, create one, reserve its prompt) on a shuffled pool: after every
    phase each live sequence holds the length and the pages the allocator
    model hands out for the same calls, and the free count agrees."""
    num_pages, P = 40, 16
    cfg = kd.make_config(1, 8, 8, 64, num_pages, 6, 8)
    h = kd.kv_cache_create(cfg)
    perm = np.random.default_rng(17).permutation(num_pages)
    kd.kv_cache_set_page_order(h, perm)
    m = PagePoolModel(num_pages, P, 6, 8)
    m.set_page_order(perm)
    batch = []
    for n in (5, 16, 30, 47):
        s_ = kd.kv_seq_create(h)
        assert s_ == m.seq_create()
        kd.kv_seq_reserve(h, s_, n)
        m.seq_reserve(s_, n)
        batch.append(s_)
    kd.kv_cache_device_steps(h, 6)

    def check():
        st = kd.kv_cache_query(h)
        assert st.free_pages == len(m.free) and st.pages_in_use == num_pages - len(m.free)
        for s_ in batch:
            assert kd.kv_seq_info(h, s_) == (m.lens[s_], m.pages[s_]), s_

    for phase in range(3):
        ids = torch.tensor(batch, dtype=torch.int32, device="cuda")
        for _ in range(7):
            kd.kv_begin_step_device(h, len(batch), ids)
            m.begin_step(batch)
        torch.cuda.synchronize()
        check()
        victim = batch[(phase + 1) % len(batch)]
        kd.kv_seq_free(h, victim)
        m.seq_free(victim)
        new = kd.kv_seq_create(h)
        assert new == m.seq_create()
        kd.kv_seq_reserve(h, new, 20)
        m.seq_reserve(new, 20)
        batch[batch.index(victim)] = new
        check()
    kd.kv_cache_destroy(h)


def test_host_step_cannot_move_buffers_under_device_steps(kvlib):
    """Device steps reserve plan buffers (captured graphs point at them); a
    host-planned step that needs more fails with KVC_ERR_INVALID and changes
    nothing, and works once device steps are disabled."""
    cfg = kd.make_config(1, 8, 8, 64, 600, 4, 128)
    h = kd.kv_cache_create(cfg)
    seqs = [kd.kv_seq_create(h) for _ in range(4)]
    for s_ in seqs:
        kd.kv_seq_reserve(h, s_, 1900)
    kd.kv_cache_set_split_pages(h, 4)
    kd.kv_cache_device_steps(h, 2)          # room for 2 rows x 32 items
    before = [kd.kv_seq_info(h, s_) for s_ in seqs]
    with pytest.raises(kd.KVDecodeError) as ei:
        kd.kv_begin_step(h, seqs)           # 4 rows x 30 items
    assert ei.value.code == kd.KVC_ERR_INVALID and "disable device steps" in str(ei.value)
    assert [kd.kv_seq_info(h, s_) for s_ in seqs] == before
    kd.kv_cache_device_steps(h, 2, False)
    kd.kv_begin_step(h, seqs)
    assert [kd.kv_seq_info(h, s_)[0] for s_ in seqs] == [1901] * 4
    kd.kv_cache_destroy(h)


def test_batch_beyond_one_block_device_and_host_steps(kvlib):
    """1100 rows: the step kernels plan and copy page lists in two chunks of
    1024 rows (the host step also takes two launches); device and host steps
    give bit-identical outputs, and rows from both chunks match the oracle."""
    rng = np.random.default_rng(11)
    lens = [int(x) for x in rng.integers(0, 90, 1100)]
    cfg = wl.custom("wide_batch", 1, 8, 2, 64, 1100, lens=lens, seed=19, page_order="shuffled")
    keep = [0, 1, 500, 1023, 1024, 1025, 1099]
    a = Tracked(cfg, extra_tokens=6, split_pages=SPLIT, keep_host=True, keep_rows=keep)
    b = Tracked(cfg, extra_tokens=6, split_pages=SPLIT, keep_host=False)
    kd.kv_cache_device_steps(b.sess.h, cfg.batch)
    ids = torch.tensor(b.sess.seq_ids, dtype=torch.int32, device="cuda")
    for step in range(3):
        a.begin_step()
        kd.kv_begin_step_device(b.sess.h, cfg.batch, ids)
        b.step += 1
        b.sess.lens += 1
        oa, q, _, _ = a.run_layer(0, fused=True)
        ob, _, _, _ = b.run_layer(0, fused=True)
        torch.cuda.synchronize()
        assert torch.equal(oa, ob), step
        ref, vmax = a.oracle(0, q, rows=keep)
        assert_close(bf16_to_f64(ob)[keep], ref, vmax, gqa=True, what=step)
    a.close()
    b.close()


def test_layer_graph_captured_after_another_replays_as_fast(kvlib):
    """Two graphs of the same fused layers, captured one after the other, each
    replayed after a graph of the device-side step: the second graph's first
    layer must not wait for an announcement from the first graph's last
    layer, which at replay is not its predecessor (its time stays within 2x
    of the first graph's; a missed announcement would add its 0.5 ms wait)."""
    cfg = wl.custom("twographs", 4, 8, 8, 64, 4, lens=[300, 17, 900, 64], seed=21)
    t = Tracked(cfg, keep_host=False, extra_tokens=200)
    h = t.sess.h
    B, L = cfg.batch, cfg.num_layers
    stream = torch.cuda.Stream()
    ids = torch.tensor(t.sess.seq_ids, dtype=torch.int32, device="cuda")
    kd.kv_cache_device_steps(h, B, True, stream)
    ins = [wl.step_inputs(cfg, 0, l, "cuda") for l in range(L)]
    outs = [torch.empty_like(x[0]) for x in ins]

    def layers():
        for l in range(L):
            kd.decode_attention_append(h, l, B, ins[l][0], ins[l][1], ins[l][2], outs[l], 0.0, stream)

    with torch.cuda.stream(stream):
        kd.kv_begin_step_device(h, B, ids, stream)
        layers()
    stream.synchronize()
    g_step, g_a, g_b = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_step, stream=stream):
        kd.kv_begin_step_device(h, B, ids, stream)
    with torch.cuda.graph(g_a, stream=stream):
        layers()
    with torch.cuda.graph(g_b, stream=stream):
        layers()

    def timed(g):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        with torch.cuda.stream(stream):
            for _ in range(3):
                g_step.replay()
                g.replay()
            ev[0].record(stream)
            for _ in range(10):
                g_step.replay()
                g.replay()
            ev[1].record(stream)
        stream.synchronize()
        return ev[0].elapsed_time(ev[1]) / 10

    ta, tb = timed(g_a), timed(g_b)
    assert tb < 2 * ta + 0.05, (ta, tb)
    st = kd.kv_cache_query(h)
    assert st.device_error == 0
    t.close()
