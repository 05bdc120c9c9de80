"""Pins of the float64 oracle against things other than itself: values the
paper prints (tests/golden), closed forms, invariants of the definition,
library routines (torch SDPA, scipy softmax, torch's bf16 widening) and a
pure-Python brute force on tiny inputs.  CPU only."""
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import PagePoolModel, OutOfPages

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf16_bits(x: torch.Tensor) -> np.ndarray:
    return x.to(torch.bfloat16).contiguous().view(torch.int16).numpy().view(np.uint16)


def rand_bits(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return bf16_bits(torch.randn(*shape, generator=g) * scale)


# --------------------------------------------------------------------------
# bf16 widening
# --------------------------------------------------------------------------
def test_bf16_widening_matches_torch_for_every_bit_pattern(oracle_lib):
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = oracle.bf16_to_f64(bits)
    ref = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).to(torch.float64).numpy()
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])
    # spot values fixed by the format: 0x3F80 = 1.0, 0xC000 = -2.0, 0x0001 = 2^-133
    assert oracle.bf16_to_f64(np.array([0x3F80, 0xC000, 0x0001], np.uint16)).tolist() == [1.0, -2.0, 2.0 ** -133]


# --------------------------------------------------------------------------
# Eq. 1 footprint against the values the paper prints
# --------------------------------------------------------------------------
def _golden_rows(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                rows.append(line.split())
    return rows


def test_eq1_matches_printed_values():
    rows = _golden_rows("eq1_footprint.txt")
    assert len(rows) == 4
    for label, L, nkv, dh, s, b, val, unit, _where in rows:
        got = oracle.kv_bytes_eq1(int(L), int(nkv), int(dh), int(s), int(b))
        val = float(val)
        if unit == "MiB":
            assert got == val * 2 ** 20, label          # exact: the printed M are MiB
        elif unit == "MB_approx":
            assert abs(got / 2 ** 20 - val) / val < 0.01, label
        elif unit == "GB_approx":
            assert abs(got / 2 ** 30 - val) / val < 0.02, label
        else:
            raise AssertionError(unit)
    # the worked example's exact byte count
    assert oracle.kv_bytes_eq1(32, 32, 128, 704, 2) == 369_098_752


def test_paged_footprint_equals_eq1_on_page_multiples_and_rounds_up_otherwise():
    assert oracle.kv_bytes_paged(32, 32, 128, 16, [704]) == oracle.kv_bytes_eq1(32, 32, 128, 704)
    # 705 tokens hold 45 pages = 720 token slots
    assert oracle.kv_bytes_paged(32, 32, 128, 16, [705]) == oracle.kv_bytes_eq1(32, 32, 128, 720)
    assert oracle.kv_bytes_paged(28, 4, 128, 16, [1, 16, 17]) == oracle.kv_bytes_eq1(28, 4, 128, 16 * 4)


# --------------------------------------------------------------------------
# attention: closed forms and invariants
# --------------------------------------------------------------------------
def test_single_token_context_returns_v(oracle_lib):
    q = rand_bits((3, 4, 64), 1)
    k = rand_bits((3, 2, 64), 2)
    v = rand_bits((3, 2, 64), 3)
    out = oracle.decode_attention(q, [1, 1, 1], k, v)
    vv = oracle.bf16_to_f64(v)
    for b in range(3):
        for h in range(4):
            assert np.array_equal(out[b, h], vv[b, h // 2])


def test_identical_keys_give_mean_of_v(oracle_lib):
    n, d = 37, 128
    q = rand_bits((1, 1, d), 4)
    k1 = rand_bits((1, 1, d), 5)
    k = np.repeat(k1, n, axis=0)
    v = rand_bits((n, 1, d), 6)
    out = oracle.decode_attention(q, [n], k, v)
    mean = oracle.bf16_to_f64(v)[:, 0, :].mean(axis=0)
    np.testing.assert_allclose(out[0, 0], mean, rtol=1e-13, atol=1e-15)


def test_zero_query_gives_mean_of_v(oracle_lib):
    n, d = 50, 64
    q = np.zeros((1, 2, d), np.uint16)
    k = rand_bits((n, 2, d), 7)
    v = rand_bits((n, 2, d), 8)
    out = oracle.decode_attention(q, [n], k, v)
    mean = oracle.bf16_to_f64(v).mean(axis=0)
    np.testing.assert_allclose(out[0], mean, rtol=1e-13, atol=1e-15)


def test_weights_sum_to_one(oracle_lib):
    lens = [1, 5, 97, 300]
    q = rand_bits((4, 8, 64), 9, 3.0)
    k = rand_bits((sum(lens), 8, 64), 10, 3.0)
    v = rand_bits((sum(lens), 8, 64), 11)
    _, ws = oracle.decode_attention(q, lens, k, v, return_wsum=True)
    assert np.all(np.abs(ws - 1.0) < 1e-12)


def test_one_hot_query_selects_that_value(oracle_lib):
    n, d = 40, 64
    k = np.zeros((n, 1, d), np.uint16)
    hot = 17
    kk = np.zeros((n, 1, d), np.float32)
    for t in range(n):
        kk[t, 0, t % d] = 1.0
    k = bf16_bits(torch.from_numpy(kk))
    qq = np.zeros((1, 1, d), np.float32)
    qq[0, 0, hot] = 1000.0   # score gap 1000/sqrt(64) = 125 -> other weights < e^-125
    q = bf16_bits(torch.from_numpy(qq))
    v = rand_bits((n, 1, d), 12)
    out = oracle.decode_attention(q, [n], k, v)
    np.testing.assert_allclose(out[0, 0], oracle.bf16_to_f64(v)[hot, 0], rtol=1e-12, atol=1e-40)


def _sdpa_reference(q, lens, k, v, scale=None):
    """torch SDPA in float64 with K/V heads repeated to the query heads."""
    qd = torch.from_numpy(oracle.bf16_to_f64(q))
    kd = torch.from_numpy(oracle.bf16_to_f64(k))
    vd = torch.from_numpy(oracle.bf16_to_f64(v))
    B, Hq, d = qd.shape
    G = Hq // kd.shape[1]
    outs = []
    off = 0
    for b, n in enumerate(lens):
        kb = kd[off:off + n].permute(1, 0, 2).repeat_interleave(G, dim=0)   # [Hq, n, d]
        vb = vd[off:off + n].permute(1, 0, 2).repeat_interleave(G, dim=0)
        qb = qd[b].unsqueeze(1)                                            # [Hq, 1, d]
        o = torch.nn.functional.scaled_dot_product_attention(qb, kb, vb, scale=scale)
        outs.append(o[:, 0, :])
        off += n
    return torch.stack(outs).numpy()


@pytest.mark.parametrize("Hq,Hkv,d", [(8, 8, 64), (28, 4, 128), (6, 2, 32), (7, 1, 16)])
def test_matches_torch_sdpa_float64(oracle_lib, Hq, Hkv, d):
    lens = [1, 3, 17, 64, 129]
    q = rand_bits((len(lens), Hq, d), 100 + Hq, 2.0)
    k = rand_bits((sum(lens), Hkv, d), 200 + Hq, 2.0)
    v = rand_bits((sum(lens), Hkv, d), 300 + Hq)
    ours = oracle.decode_attention(q, lens, k, v)
    ref = _sdpa_reference(q, lens, k, v)
    np.testing.assert_allclose(ours, ref, rtol=1e-12, atol=1e-13)
    # a non-default scale is honoured the same way
    ours2 = oracle.decode_attention(q, lens, k, v, scale=0.3)
    ref2 = _sdpa_reference(q, lens, k, v, scale=0.3)
    np.testing.assert_allclose(ours2, ref2, rtol=1e-12, atol=1e-13)


def test_matches_scipy_softmax_einsum(oracle_lib):
    from scipy.special import softmax
    n, Hq, Hkv, d = 70, 12, 3, 64
    q = rand_bits((1, Hq, d), 41, 2.0)
    k = rand_bits((n, Hkv, d), 42, 2.0)
    v = rand_bits((n, Hkv, d), 43)
    qd, kd, vd = (oracle.bf16_to_f64(x) for x in (q, k, v))
    G = Hq // Hkv
    heads = np.arange(Hq) // G
    s = np.einsum("hd,thd->ht", qd[0], kd[:, heads, :]) / math.sqrt(d)
    ref = np.einsum("ht,thd->hd", softmax(s, axis=1), vd[:, heads, :])
    np.testing.assert_allclose(oracle.decode_attention(q, [n], k, v)[0], ref, rtol=1e-12, atol=1e-13)


def test_brute_force_pure_python_tiny(oracle_lib):
    """Independent enumeration with math.exp on a tiny GQA case."""
    lens = [2, 5]
    Hq, Hkv, d = 4, 2, 8
    q = rand_bits((2, Hq, d), 51, 2.0)
    k = rand_bits((7, Hkv, d), 52, 2.0)
    v = rand_bits((7, Hkv, d), 53)
    qd, kd, vd = (oracle.bf16_to_f64(x).tolist() for x in (q, k, v))
    ours = oracle.decode_attention(q, lens, k, v)
    off = 0
    for b, n in enumerate(lens):
        for h in range(Hq):
            g = h // (Hq // Hkv)
            sc = [sum(qd[b][h][i] * kd[off + t][g][i] for i in range(d)) / math.sqrt(d) for t in range(n)]
            e = [math.exp(x - max(sc)) for x in sc]
            z = sum(e)
            for i in range(d):
                ref = sum(e[t] / z * vd[off + t][g][i] for t in range(n))
                assert abs(ours[b, h, i] - ref) <= 1e-12 * (1 + abs(ref))
        off += n


def test_gqa_equals_mha_on_repeated_kv_heads(oracle_lib):
    """Grouping g = h / G: GQA on H_kv heads is MHA on K/V heads repeated G
    times (consecutive query heads share a KV head)."""
    lens = [33, 80]
    Hq, Hkv, d = 28, 4, 64
    q = rand_bits((2, Hq, d), 61)
    k = rand_bits((sum(lens), Hkv, d), 62)
    v = rand_bits((sum(lens), Hkv, d), 63)
    gqa = oracle.decode_attention(q, lens, k, v)
    mha = oracle.decode_attention(q, lens, np.repeat(k, 7, axis=1), np.repeat(v, 7, axis=1))
    assert np.array_equal(gqa, mha)


# --------------------------------------------------------------------------
# paged layout: scatter / gather and page-order invariance
# --------------------------------------------------------------------------
def _paged_pool(num_pages, Hkv, P, d, fill=0xFFFF):
    return np.full((num_pages, Hkv, P, d), fill, dtype=np.uint16)


def test_scatter_gather_roundtrip_and_touches_only_its_slots(oracle_lib):
    num_pages, Hkv, P, d = 12, 3, 4, 8
    rng = np.random.default_rng(3)
    perm = rng.permutation(num_pages).astype(np.int32)
    n = 10
    row = perm[:3]
    x = rand_bits((n, Hkv, d), 71)
    pool = _paged_pool(num_pages, Hkv, P, d)
    oracle.kv_scatter(pool, row, 0, x, P)
    assert np.array_equal(oracle.kv_gather(pool, row, 0, n), x)
    # exactly n * Hkv * d elements changed, all inside the row's pages
    changed = pool != 0xFFFF
    assert int(changed.sum()) == int((x != 0xFFFF).sum())
    assert not changed[np.setdiff1d(np.arange(num_pages), row)].any()
    # library reading of the same layout: [pages, Hkv, P, d] -> [pages*P, Hkv, d]
    flat = pool.transpose(0, 2, 1, 3).reshape(num_pages * P, Hkv, d)
    phys = (np.repeat(row, P) * P + np.tile(np.arange(P), len(row)))[:n]
    assert np.array_equal(flat[phys], x)
    # an append at position n writes slot n % P of page row[n // P]
    y = rand_bits((1, Hkv, d), 72)
    oracle.kv_scatter(pool, row, n, y, P)
    assert np.array_equal(pool.transpose(0, 2, 1, 3)[row[n // P], n % P], y[0])
    with pytest.raises(ValueError):
        oracle.kv_scatter(pool, np.array([num_pages], np.int32), 0, y, P)


def test_paged_attention_is_invariant_to_physical_page_order(oracle_lib):
    P, Hq, Hkv, d = 16, 14, 2, 64
    lens = [1, 16, 17, 95]
    B = len(lens)
    q = rand_bits((B, Hq, d), 81)
    k = rand_bits((sum(lens), Hkv, d), 82)
    v = rand_bits((sum(lens), Hkv, d), 83)
    logical = oracle.decode_attention(q, lens, k, v)
    npages = [(n + P - 1) // P for n in lens]
    total = sum(npages) + 3
    outs = []
    for seed in (0, 1, 2):
        perm = np.random.default_rng(seed).permutation(total).astype(np.int32)
        kp, vp = _paged_pool(total, Hkv, P, d, 0x7FC0), _paged_pool(total, Hkv, P, d, 0x7FC0)  # NaN filler
        pt = np.full((B, max(npages)), -1, np.int32)
        used = 0
        off = 0
        for b, n in enumerate(lens):
            pt[b, :npages[b]] = perm[used:used + npages[b]]
            used += npages[b]
            oracle.kv_scatter(kp, pt[b], 0, k[off:off + n], P)
            oracle.kv_scatter(vp, pt[b], 0, v[off:off + n], P)
            off += n
        outs.append(oracle.decode_attention_paged(q, lens, pt, kp, vp))
    for o in outs:
        assert np.array_equal(o, logical)   # bit-identical: same values, same order of sums


# --------------------------------------------------------------------------
# allocator model
# --------------------------------------------------------------------------
def test_allocator_model_hand_worked_example():
    lines = []
    with open(os.path.join(GOLDEN, "allocator_lazy_example.txt")) as f:
        for line in f:
            s = line.split("#")[0].strip()
            if s:
                lines.append(s.split())
    m = PagePoolModel(8, 4, 4, 4)
    m.set_page_order([5, 2, 7, 0, 3, 6, 1, 4])
    created = []
    for op, *args in lines:
        if op == "create":
            created.append(m.seq_create())
        elif op == "reserve":
            m.seq_reserve(int(args[0]), int(args[1]))
        elif op == "step":
            m.begin_step([int(a) for a in args])
        elif op == "free":
            m.seq_free(int(args[0]))
        elif op == "expect":
            seq, ln, pages = int(args[0]), int(args[1]), [int(x) for x in args[2].split(",")]
            assert m.lens[seq] == ln and m.pages[seq] == pages, (op, args)
        elif op == "free_pages":
            assert len(m.free) == int(args[0])
    assert created == [0, 1, 0]


def test_allocator_model_properties():
    P, num_pages = 16, 200
    m = PagePoolModel(num_pages, P, 16, 64)
    rng = np.random.default_rng(5)
    m.set_page_order(rng.permutation(num_pages))
    live = []
    for it in range(300):
        r = rng.random()
        if r < 0.2 and len(live) < 16:
            live.append(m.seq_create())
        elif r < 0.3 and live:
            s = live.pop(int(rng.integers(len(live))))
            m.seq_free(s)
        elif live:
            s = live[int(rng.integers(len(live)))]
            n = int(rng.integers(0, 40))
            before = (dict(m.lens), {k: list(v) for k, v in m.pages.items()}, list(m.free))
            try:
                m.seq_reserve(s, n)
            except OutOfPages:
                assert (m.lens, m.pages, m.free) == before      # all or nothing
            except ValueError:
                assert (m.lens, m.pages, m.free) == before
        # invariants: ceil(len/P) pages per sequence, all distinct, pool conserved
        used = [p for s in m.pages for p in m.pages[s]]
        assert len(used) == len(set(used))
        assert sorted(used + m.free) == list(range(num_pages))
        for s in m.lens:
            assert len(m.pages[s]) == (m.lens[s] + P - 1) // P


def test_allocator_model_oom_and_row_limit():
    m = PagePoolModel(2, 4, 2, 2)
    a = m.seq_create()
    m.seq_reserve(a, 8)
    with pytest.raises(ValueError):
        m.seq_reserve(a, 1)        # would need a third page in a 2-wide row
    b = m.seq_create()
    with pytest.raises(OutOfPages):
        m.seq_reserve(b, 1)
    with pytest.raises(OutOfPages):
        m.begin_step([b])
    assert m.lens[b] == 0 and m.pages[b] == []
