"""Failure detection on the GPU without faulting it: a device-side wait that
runs out reports a status and leaves the context usable; a corrupt page id
is recorded in the error word and replaced by a valid page (no fault)."""
import time

import numpy as np
import pytest
import torch

from paper_2603_12707_gb300 import kvdecode as kd
from paper_2603_12707_gb300 import workloads as wl

from _gpu_common import Tracked, bf16_to_f64

pytestmark = pytest.mark.gpu


def test_bounded_wait_gives_up_and_context_stays_usable(kvlib):
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    t0 = time.perf_counter()
    kd.kv_selftest_wait_timeout(50_000_000, status)   # 50 ms on a barrier nothing completes
    torch.cuda.synchronize()
    assert time.perf_counter() - t0 < 5.0
    assert int(status.item()) == 1
    # the context still runs work
    cfg = wl.custom("after_timeout", 1, 8, 8, 64, 2, lens=[20, 40], seed=2)
    t = Tracked(cfg, keep_host=True)
    t.begin_step()
    out, q, _, _ = t.run_layer(0)
    torch.cuda.synchronize()
    ref, _ = t.oracle(0, q)
    assert np.abs(bf16_to_f64(out) - ref).max() < 2e-2
    t.close()


def test_corrupt_page_id_is_reported_not_faulted(kvlib):
    cfg = wl.custom("badpage", 1, 28, 4, 128, 3, lens=[300, 47, 100], seed=8)
    t = Tracked(cfg, keep_host=False)
    sess = t.sess
    t.begin_step()
    _, q, _, _ = t.run_layer(0)
    torch.cuda.synchronize()
    pt = np.full((cfg.batch, sess.max_pages), -1, np.int32)
    lens = []
    for b, seq in enumerate(sess.seq_ids):
        ln, pages = kd.kv_seq_info(sess.h, seq)
        pt[b, :len(pages)] = pages
        lens.append(ln)
    kp, vp = kd.kv_cache_pool(sess.h, 0)
    out = torch.empty_like(q)
    for bad in (-5, sess.num_pages + 3):
        pt_bad = pt.copy()
        pt_bad[0, 1] = bad
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        kd.decode_attention_noalloc(kp, vp, sess.num_pages, 28, 4, 128, torch.from_numpy(pt_bad).cuda(),
                                    sess.max_pages, lens, q, out, 0.0, err)
        torch.cuda.synchronize()
        assert int(err.item()) & kd.KVC_DEVERR_PAGE_RANGE
        assert torch.isfinite(out.float()).all()
    # a clean table reports nothing
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    kd.decode_attention_noalloc(kp, vp, sess.num_pages, 28, 4, 128, torch.from_numpy(pt).cuda(), sess.max_pages,
                                lens, q, out, 0.0, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    t.close()
