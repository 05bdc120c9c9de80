"""decode_attention_noalloc, the entry point for callers that may not
allocate device memory while serving (a plugin held to a memory budget fixed
at build time, a runtime whose device memory belongs to another framework's
allocator).  It runs on a 16 MiB static scratch array instead of cache-owned
buffers; here its output is checked against decode_attention's on the same
cache contents, on two calls in a row (the second reuses the scratch the
first left behind).  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

from paper_2603_12707_gb300 import kvdecode as kd
from paper_2603_12707_gb300 import workloads as wl

from _gpu_common import Tracked, bf16_to_f64, u16

pytestmark = pytest.mark.gpu


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
])
def test_noalloc_matches_decode_attention_on_two_calls(kvlib, Hq, Hkv, d, lens):
    cfg = wl.custom("noalloc", 2, Hq, Hkv, d, len(lens), lens=lens, seed=17 + Hq, page_order="shuffled")
    t = Tracked(cfg, keep_host=False)
    sess = t.sess
    t.begin_step()
    out_ref, q, _, _ = t.run_layer(1)
    pt = _page_table(sess)
    attended = [int(n) for n in sess.lens]
    kp, vp = kd.kv_cache_pool(sess.h, 1)
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
        _close(bf16_to_f64(out), bf16_to_f64(out_ref), vmax, Hq > Hkv)
    assert int(err.item()) == 0
    t.close()


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
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 128, pt, sess.max_pages, [1] * 1025, q, out)
    assert ei.value.code == kd.KVC_ERR_INVALID
    with pytest.raises(kd.KVDecodeError) as ei:      # a length beyond the page-table row
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 128, pt, sess.max_pages,
                                    [sess.max_pages * 16 + 1, 1], q, out)
    assert ei.value.code == kd.KVC_ERR_INVALID
    with pytest.raises(kd.KVDecodeError) as ei:      # head_dim outside {64, 128}
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 32, 32, 96, pt, sess.max_pages, [4, 4], q, out)
    assert ei.value.code == kd.KVC_ERR_UNSUPPORTED
    t.close()
