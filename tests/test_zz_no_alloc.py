"""decode_attention_noalloc, the entry point for callers that may not
allocate device memory while serving (a plugin held to a memory budget fixed
at build time, a runtime whose device memory belongs to another framework's
allocator).  It runs on a 16 MiB static scratch array instead of cache-owned
buffers.  Checked here: its output against decode_attention's on the same
cache contents and against the float64 oracle reading the same pools through
the same page table, with NaN / Inf patterns in every pool slot no row holds,
on two calls in a row (the second reuses the scratch the first left behind); a batch whose plan only fits the scratch after the item
size has doubled; a batch that never fits (KVC_ERR_UNSUPPORTED); argument
checks.  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

import oracle
from paper_2603_12707_gb300 import kvdecode as kd
from paper_2603_12707_gb300 import workloads as wl

from _gpu_common import Tracked, assert_close, bf16_to_f64, device_pool, poison_unused_slots, u16

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 16 << 20


def _page_table(sess):
    pt = np.full((sess.cfg.batch, sess.max_pages), -1, np.int32)
    for b, seq in enumerate(sess.seq_ids):
        _, pages = kd.kv_seq_info(sess.h, seq)
        pt[b, :len(pages)] = pages
    return torch.from_numpy(pt).cuda()


def _close(got, ref, vmax, gqa):
    # both outputs are within the parity bound of the exact result, so they
    # differ by at most twice that bound
    err = np.abs(got - ref)
    assert err.max() <= 2e-2 and err.mean() <= 2e-3
    w = (2.0 ** -8 if gqa else 0.0) + 1e-5
    assert (err <= 2.0 ** -7 * np.abs(ref) + 2 * w * vmax[:, None, None]).all()


@pytest.mark.parametrize("Hq,Hkv,d,lens", [
    (32, 32, 128, [700, 1, 16, 17, 1300, 95]),
    (28, 4, 128, [2048, 300, 33, 5000]),
    (8, 8, 64, [96, 96, 96, 96]),
    (16, 2, 64, [1, 250, 31, 700, 16]),
])
def test_noalloc_matches_decode_attention_and_oracle_on_two_calls(kvlib, Hq, Hkv, d, lens):
    cfg = wl.custom("noalloc", 2, Hq, Hkv, d, len(lens), lens=lens, seed=17 + Hq, page_order="shuffled")
    t = Tracked(cfg, keep_host=False)
    sess = t.sess
    poison_unused_slots(sess)      # NaN / Inf in every slot no row holds
    t.begin_step()
    out_ref, q, _, _ = t.run_layer(1)
    pt = _page_table(sess)
    attended = [int(n) for n in sess.lens]
    kp, vp = kd.kv_cache_pool(sess.h, 1)
    # the pools' bytes (the prefix and this step's appended token) for the oracle
    k_host, v_host = device_pool(sess, 1)
    pt_host = pt.cpu().numpy()
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    vmax = np.array([np.abs(bf16_to_f64(wl.kv_block(cfg, 1, b, max(1, n), "v", "cuda"))).max() + 1e-30
                     for b, n in enumerate(sess.lens0)])
    vmax = np.maximum(vmax, 4.0 * cfg.kv_scale)
    for call in range(2):
        if call == 1:
            # a different query on the same cache, through both entry points
            q = wl.step_inputs(cfg, 7, 1, "cuda")[0]
            out_ref = torch.empty_like(q)
            sess.attend(1, q, out_ref)
        out = torch.full_like(q, float("nan"))
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, Hq, Hkv, d, pt, sess.max_pages, attended, q, out,
                                    0.0, err)
        torch.cuda.synchronize()
        got = bf16_to_f64(out)
        _close(got, bf16_to_f64(out_ref), vmax, Hq > Hkv)
        exact = oracle.decode_attention_paged(u16(q), attended, pt_host, k_host, v_host)
        assert_close(got, exact, vmax, Hq > Hkv, f"noalloc call {call}")
    assert int(err.item()) == 0
    t.close()


def _scratch_bytes(lens, T, Hkv, G, d, cap=32):
    """Scratch the entry point needs at item size T (the layout it documents:
    plan entries of 32 B, each entry's page ids, and (o, m, l) partials for
    rows cut into several items), each part rounded up to 256 B."""
    r = lambda x: (x + 255) // 256 * 256
    entries, split_items, stride = 0, 0, 1
    for n in lens:
        np_ = (n + 15) // 16
        tb = max(T, (np_ + cap - 1) // cap)
        nch = (np_ + tb - 1) // tb
        entries += nch
        split_items += nch if nch > 1 else 0
        stride = max(stride, (np_ + nch - 1) // nch)
    slots = split_items * Hkv
    off = r(entries * 32)
    off = r(off + entries * stride * 4)
    off = r(off + slots * G * d * 4)
    off = r(off + slots * G * 8)
    off = r(off + len(lens) * 8)
    return r(off + 12)


def _shared_pool(num_pages, Hkv, d, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    k = (torch.randn((num_pages, Hkv, 16, d), generator=g, device="cuda") / d ** 0.5).to(torch.bfloat16)
    v = torch.randn((num_pages, Hkv, 16, d), generator=g, device="cuda").to(torch.bfloat16)
    return k, v


def test_noalloc_item_size_doubles_until_the_plan_fits(kvlib):
    """1024 rows of 6200 .. 8192 tokens over a 64-page pool that every row's
    page list draws from (the caller owns the page table, so rows may share
    pages).  At the first item size (128 pages: the usual target is far above
    it for this batch) each row is cut into 4 items whose partials need more
    than 16 MiB; at 256 pages each row has 2 items and the plan fits, so the
    merge pass still runs.  Sampled rows against the oracle."""
    Hq = Hkv = 8
    d, batch, num_pages = 128, 1024, 64
    rng = np.random.default_rng(5)
    lens = rng.integers(6200, 8193, size=batch).astype(np.int32)
    lens[0], lens[1] = 8192, 6200
    max_pages = 512
    assert _scratch_bytes(lens, 128, Hkv, 1, d) > SCRATCH_BYTES
    assert _scratch_bytes(lens, 256, Hkv, 1, d) <= SCRATCH_BYTES
    pt = rng.integers(0, num_pages, size=(batch, max_pages)).astype(np.int32)
    kp, vp = _shared_pool(num_pages, Hkv, d, 41)
    pt_dev = torch.from_numpy(pt).cuda()
    g = torch.Generator(device="cuda").manual_seed(43)
    q = torch.randn((batch, Hq, d), generator=g, device="cuda").to(torch.bfloat16)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    k_host, v_host = u16(kp), u16(vp)
    vmax = np.full(batch, np.abs(bf16_to_f64(vp)).max())
    rows = [0, 1, 2, 511, 1022, 1023] + rng.choice(np.arange(3, 1022), 6, replace=False).tolist()
    prev = None
    for call in range(2):
        out = torch.full_like(q, float("nan"))
        kd.decode_attention_noalloc(kp, vp, num_pages, Hq, Hkv, d, pt_dev, max_pages, lens.tolist(), q, out,
                                    0.0, err)
        torch.cuda.synchronize()
        got = bf16_to_f64(out)
        assert np.isfinite(got).all()
        exact = oracle.decode_attention_paged(u16(q)[rows], lens[rows], pt[rows], k_host, v_host)
        assert_close(got[rows], exact, vmax[rows], False, f"doubled items, call {call}")
        if prev is not None:
            assert np.array_equal(got, prev)   # same inputs, same plan: same bits
        prev = got
    assert int(err.item()) == 0


def test_noalloc_reports_a_plan_that_never_fits(kvlib):
    """1024 rows of 32768 tokens with 32 KV heads: even at the largest item
    size (1024 pages) every row has 2 items, whose partials need 34 MB.  The
    call returns KVC_ERR_UNSUPPORTED before enqueueing anything."""
    Hq = Hkv = 32
    d, batch, num_pages, max_pages = 128, 1024, 16, 2048
    lens = [32768] * batch
    assert _scratch_bytes(lens, 1024, Hkv, 1, d) > SCRATCH_BYTES
    kp, vp = _shared_pool(num_pages, Hkv, d, 7)
    pt = torch.zeros((batch, max_pages), dtype=torch.int32, device="cuda")
    q = torch.zeros((batch, Hq, d), dtype=torch.bfloat16, device="cuda")
    out = torch.full_like(q, 7.0)
    with pytest.raises(kd.KVDecodeError) as ei:
        kd.decode_attention_noalloc(kp, vp, num_pages, Hq, Hkv, d, pt, max_pages, lens, q, out)
    assert ei.value.code == kd.KVC_ERR_UNSUPPORTED
    assert "16 MiB" in str(ei.value)
    torch.cuda.synchronize()
    assert bool((out == 7.0).all())    # nothing ran


def test_noalloc_rejects_what_does_not_fit(kvlib):
    cfg = wl.custom("noalloc_err", 1, 32, 32, 128, 2, lens=[40, 40], seed=3)
    t = Tracked(cfg, keep_host=False)
    sess = t.sess
    t.begin_step()
    _, q, _, _ = t.run_layer(0)
    kp, vp = kd.kv_cache_pool(sess.h, 0)
    pt = _page_table(sess)
    out = torch.empty_like(q)
    with pytest.raises(kd.KVDecodeError) as ei:      # batch above 1024
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 128, pt.data_ptr(), sess.max_pages,
                                    [1] * 1025, q.data_ptr(), out.data_ptr())
    assert ei.value.code == kd.KVC_ERR_INVALID
    with pytest.raises(kd.KVDecodeError) as ei:      # a length beyond the page-table row
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 128, pt, sess.max_pages,
                                    [sess.max_pages * 16 + 1, 1], q, out)
    assert ei.value.code == kd.KVC_ERR_INVALID
    with pytest.raises(kd.KVDecodeError) as ei:      # head_dim outside {64, 128}
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 96, pt.data_ptr(), sess.max_pages, [4, 4],
                                    q.data_ptr(), out.data_ptr())
    assert ei.value.code == kd.KVC_ERR_UNSUPPORTED
    # tensors the binding can see are checked before the call
    with pytest.raises(ValueError):                  # page table of the wrong type
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 128, pt.long(), sess.max_pages, [4, 4], q, out)
    with pytest.raises(ValueError):                  # page table shorter than max_pages
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 128, pt[:, :1].contiguous(), sess.max_pages,
                                    [4, 4], q, out)
    with pytest.raises(ValueError):                  # q with a row missing
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 128, pt, sess.max_pages, [4, 4], q[:1], out)
    t.close()

