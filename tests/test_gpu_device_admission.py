"""Admitting and closing sequences while device-side steps replay from a
CUDA graph, with no host synchronisation (lazy allocation at prefill entry,
Sec. 5.4 "Lazy KV Cache Allocation").

One stream carries everything: a bounded GPU wait first, then replayed decode
steps interleaved with sequence frees, creations, prompt reservations, packed
prefix writes and the batch's id swaps.  The event recorded right after the
wait must still be pending once the last call has returned: no call waited
for the GPU.  Afterwards the page tables equal the allocator model's for the
same calls, every output of the last step matches the float64 oracle, and the
device error word is clear.  Failures on the device path (an exhausted pool,
a write past a sequence's length) are reported through the device error bits
and change nothing."""
import time

import numpy as np
import pytest
import torch

import oracle
from oracle import PagePoolModel
from paper_2603_12707_gb300 import kvdecode as kd

from _gpu_common import assert_close, bf16_to_f64, u16

pytestmark = pytest.mark.gpu

P = 16


def _randn(shape, gen, scale=1.0):
    return (torch.randn(shape, generator=gen) * scale).to(torch.bfloat16)


@pytest.mark.parametrize("Hq,Hkv,d", [(8, 8, 64), (28, 4, 128)])
def test_admissions_and_frees_between_replayed_steps_need_no_host_sync(kvlib, Hq, Hkv, d):
    L, B, num_pages, max_seqs, max_pages = 2, 4, 96, 8, 16
    gen = torch.Generator().manual_seed(11 + Hq)
    stream = torch.cuda.Stream()
    cfg = kd.make_config(L, Hq, Hkv, d, num_pages, max_seqs, max_pages)
    h = kd.kv_cache_create(cfg, stream)
    perm = np.random.default_rng(5).permutation(num_pages)
    kd.kv_cache_set_page_order(h, perm)
    m = PagePoolModel(num_pages, P, max_seqs, max_pages)
    m.set_page_order(perm)
    kd.kv_cache_device_steps(h, B, True, stream)

    # every value is drawn up front, so the timed window only enqueues work
    prompt_lens = [37, 16, 50, 1, 29, 64, 3]
    prompts = [(_randn((L, n, Hkv, d), gen, d ** -0.5), _randn((L, n, Hkv, d), gen)) for n in prompt_lens]
    prompts_dev = [(k.cuda(), v.cuda()) for k, v in prompts]
    q = _randn((L, B, Hq, d), gen).cuda()
    kn = _randn((L, B, Hkv, d), gen, d ** -0.5).cuda()
    vn = _randn((L, B, Hkv, d), gen).cuda()
    out = torch.zeros((L, B, Hq, d), dtype=torch.bfloat16, device="cuda")
    torch.cuda.synchronize()
    kn_h, vn_h = u16(kn), u16(vn)
    tokens = {}      # sequence -> layer -> list of [Hkv, d] uint16 rows (logical order)
    next_prompt = [0]

    def admit():
        i = next_prompt[0]
        next_prompt[0] += 1
        k, v = prompts_dev[i]
        n = prompt_lens[i]
        s_ = kd.kv_seq_create(h)
        assert s_ == m.seq_create()
        kd.kv_seq_reserve(h, s_, n, stream)
        m.seq_reserve(s_, n)
        kd.kv_write_varlen(h, 0, L, [s_], [0, n], k, v, stream=stream)
        tokens[s_] = [list(u16(prompts[i][0][l])) for l in range(L)], [list(u16(prompts[i][1][l])) for l in range(L)]
        return s_

    def stepped(batch):
        m.begin_step(batch)
        for b, s_ in enumerate(batch):
            for l in range(L):
                tokens[s_][0][l].append(kn_h[l, b])
                tokens[s_][1][l].append(vn_h[l, b])

    batch = [admit() for _ in range(B)]
    ids_dev = torch.tensor(batch, dtype=torch.int32, device="cuda")

    def layers():
        for l in range(L):
            kd.decode_attention_append(h, l, B, q[l], kn[l], vn[l], out[l], 0.0, stream)

    with torch.cuda.stream(stream):                       # eager step: nothing lazy in the capture
        kd.kv_begin_step_device(h, B, ids_dev, stream)
        layers()
    stepped(batch)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        kd.kv_begin_step_device(h, B, ids_dev, stream)
        layers()
    swaps = [torch.empty(B, dtype=torch.int32).pin_memory() for _ in range(3)]
    stream.synchronize()

    # ---- the window: nothing below may wait for the GPU.  The stream is held
    # first by the library's bounded wait diagnostic (a 0.3 s wait on a
    # barrier nothing completes, which then records that it gave up).
    after_sleep = torch.cuda.Event()
    waited = torch.zeros(1, dtype=torch.int32, device="cuda")
    with torch.cuda.stream(stream):
        kd.kv_selftest_wait_timeout(300_000_000, waited, stream)
        after_sleep.record(stream)
        t0 = time.perf_counter()
        for reps, slot in ((2, 1), (3, 3), (1, 0)):
            for _ in range(reps):
                g.replay()
                stepped(batch)
            victim = batch[slot]
            kd.kv_seq_free(h, victim, stream)
            m.seq_free(victim)
            del tokens[victim]
            batch[slot] = admit()
            buf = swaps.pop()
            buf.copy_(torch.tensor(batch, dtype=torch.int32))
            ids_dev.copy_(buf, non_blocking=True)
        for _ in range(2):
            g.replay()
            stepped(batch)
        host_s = time.perf_counter() - t0
        pending = not after_sleep.query()
    assert pending, f"a call waited for the GPU (the wait had ended after {host_s:.3f} s of host calls)"
    stream.synchronize()
    assert int(waited.item()) == 1

    # ---- the state and the last step's outputs
    st = kd.kv_cache_query(h)
    assert st.device_error == 0
    assert st.free_pages == len(m.free) and st.pages_in_use == num_pages - len(m.free)
    assert st.live_seqs == len(m.lens)
    for s_ in m.lens:
        assert kd.kv_seq_info(h, s_) == (m.lens[s_], m.pages[s_]), s_
    got = bf16_to_f64(out)
    qh = u16(q)
    for l in range(L):
        lens = [len(tokens[s_][0][l]) for s_ in batch]
        assert lens == [m.lens[s_] for s_ in batch]
        K = np.concatenate([np.stack(tokens[s_][0][l]) for s_ in batch])
        V = np.concatenate([np.stack(tokens[s_][1][l]) for s_ in batch])
        ref = oracle.decode_attention(qh[l], lens, K, V)
        vmax = np.array([np.abs(oracle.bf16_to_f64(np.stack(tokens[s_][1][l]))).max() for s_ in batch])
        assert_close(got[l], ref, vmax, Hq > Hkv, f"layer {l}")
    kd.kv_cache_destroy(h)


def test_device_path_failures_are_reported_and_change_nothing(kvlib):
    """With device steps enabled, a reservation the pool cannot supply sets
    KVC_DEVERR_OOM and takes no page; a write past a sequence's length sets
    KVC_DEVERR_SEQ_RANGE and writes nothing; a reservation past the page row
    sets KVC_DEVERR_SEQ_RANGE."""
    Hq = Hkv = 8
    d, L = 64, 1
    cfg = kd.make_config(L, Hq, Hkv, d, 6, 4, 8)
    h = kd.kv_cache_create(cfg)
    kd.kv_cache_device_steps(h, 2)
    m = PagePoolModel(6, P, 4, 8)
    a = kd.kv_seq_create(h)
    assert a == m.seq_create()
    kd.kv_seq_reserve(h, a, 40)              # 3 pages
    m.seq_reserve(a, 40)
    b = kd.kv_seq_create(h)
    assert b == m.seq_create()
    kd.kv_seq_reserve(h, b, 70)              # needs 5 pages, 3 left
    torch.cuda.synchronize()
    st = kd.kv_cache_query(h, raise_on_device_error=False)
    assert st.device_error == kd.KVC_DEVERR_OOM
    assert kd.kv_seq_info(h, a) == (40, m.pages[a])
    assert kd.kv_seq_info(h, b) == (0, [])
    assert st.free_pages == 3

    h2 = kd.kv_cache_create(cfg)
    kd.kv_cache_device_steps(h2, 2)
    s_ = kd.kv_seq_create(h2)
    kd.kv_seq_reserve(h2, s_, 20)
    k = torch.full((30, Hkv, d), 3.0, dtype=torch.bfloat16, device="cuda")
    kd.kv_write_tokens(h2, 0, s_, 0, 30, k, k)     # 30 > 20: refused on the device
    kd.kv_write_varlen(h2, 0, 1, [s_], [0, 30], k[None], k[None])
    torch.cuda.synchronize()
    st = kd.kv_cache_query(h2, raise_on_device_error=False)
    assert st.device_error == kd.KVC_DEVERR_SEQ_RANGE
    back = torch.empty(20, Hkv, d, dtype=torch.bfloat16, device="cuda")
    kd.kv_read_tokens(h2, 0, s_, 0, 20, back, back)
    torch.cuda.synchronize()
    assert not bool((back == 3.0).any())           # the pool still holds its zeros

    h3 = kd.kv_cache_create(kd.make_config(L, Hq, Hkv, d, 16, 4, 8))
    kd.kv_cache_device_steps(h3, 2)
    s3 = kd.kv_seq_create(h3)
    kd.kv_seq_reserve(h3, s3, 8 * P)               # a full row
    kd.kv_seq_reserve(h3, s3, 1)                   # one past the row
    torch.cuda.synchronize()
    st = kd.kv_cache_query(h3, raise_on_device_error=False)
    assert st.device_error == kd.KVC_DEVERR_SEQ_RANGE
    assert kd.kv_seq_info(h3, s3)[0] == 8 * P
    for x in (h, h2, h3):
        kd.kv_cache_destroy(x)
