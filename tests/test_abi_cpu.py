"""CPU checks of libkvdecode.so: it loads without a GPU, exports every symbol
include/kvdecode.h declares, validates its arguments, and its lazy page
allocator (host-only mode: bookkeeping without device memory or kernels)
matches the oracle's allocator model page for page."""
import os
import re

import numpy as np
import pytest

import oracle
from oracle import PagePoolModel, OutOfPages

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kvdecode.h")


def declared_functions():
    text = open(HEADER).read()
    return re.findall(r"^KVC_API\s+(?:const\s+char\s*\*|int)\s*(\w+)\(", text, flags=re.M)


def test_header_declares_the_boundary(kvlib):
    names = declared_functions()
    for required in ("kv_cache_create", "kv_append", "decode_attention", "kv_cache_destroy"):
        assert required in names
    assert len(names) == 23


def test_library_exports_every_declared_symbol(kvlib):
    lib = kvlib.load()
    for name in declared_functions():
        assert hasattr(lib, name), name


def host_cache(kvlib, num_pages=64, max_seqs=8, max_pages=16, Hq=8, Hkv=8, d=64, L=2):
    cfg = kvlib.make_config(L, Hq, Hkv, d, num_pages, max_seqs, max_pages, flags=kvlib.KVC_FLAG_HOST_ONLY)
    return kvlib.kv_cache_create(cfg)


@pytest.mark.parametrize("field,value,code", [
    ("head_dim", 96, -5), ("page_size", 32, -5), ("num_q_heads", 72, -5),   # G = 9
    ("num_q_heads", 12, -1), ("num_pages", 0, -1), ("max_seqs", 70000, -1), ("flags", 8, -1),
    # TMA row coordinates (page * H_kv + head) * 16 and page-table indices stay below 2^31
    ("num_pages", 2**24, -1), ("max_pages_per_seq", 2**28, -1),
])
def test_create_rejects_bad_configs(kvlib, field, value, code):
    cfg = kvlib.make_config(2, 8, 8, 64, 64, 8, 16, flags=kvlib.KVC_FLAG_HOST_ONLY)
    setattr(cfg, field, value)
    with pytest.raises(kvlib.KVDecodeError) as ei:
        kvlib.kv_cache_create(cfg)
    assert ei.value.code == code


def test_data_and_attention_calls_refuse_host_only_caches(kvlib):
    h = host_cache(kvlib)
    s = kvlib.kv_seq_create(h)
    kvlib.kv_seq_reserve(h, s, 5)
    with pytest.raises(kvlib.KVDecodeError):
        kvlib.kv_write_tokens(h, 0, s, 0, 5, 16, 16)
    kvlib.kv_begin_step(h, [s])
    with pytest.raises(kvlib.KVDecodeError):
        kvlib.kv_append(h, 0, 1, 16, 16)
    with pytest.raises(kvlib.KVDecodeError):
        kvlib.decode_attention(h, 0, 1, 16, 16)
    kvlib.kv_cache_destroy(h)


def test_varlen_write_checks_its_blocks(kvlib):
    """kv_write_varlen validates every block before it touches the device:
    positions inside the reserved length, cu_seqlens starting at 0 and not
    decreasing, no two blocks on one position; a valid call on a host-only
    cache gets as far as the device check."""
    h = host_cache(kvlib)
    a, b = kvlib.kv_seq_create(h), kvlib.kv_seq_create(h)
    kvlib.kv_seq_reserve(h, a, 40)
    kvlib.kv_seq_reserve(h, b, 20)

    def code(ids, cu, fp=None, k=16, v=16):
        with pytest.raises(kvlib.KVDecodeError) as ei:
            kvlib.kv_write_varlen(h, 0, 1, ids, cu, k, v, first_pos=fp)
        return ei.value.code, kvlib.load().kv_last_error().decode()

    host_only = (kvlib.KVC_ERR_INVALID, "kv_write_varlen: cache was created host-only")
    assert code([a, b], [0, 40, 60]) == host_only
    assert code([a, a, b], [0, 10, 40, 60], fp=[0, 10, 0]) == host_only       # adjacent, no overlap
    assert code([a, a], [0, 10, 10], fp=[30, 5]) == host_only                  # an empty block is skipped
    assert "reserved length" in code([a, b], [0, 40, 61])[1]
    assert "reserved length" in code([a], [0, 5], fp=[36])[1]
    assert "cu_seqlens[0]" in code([a], [1, 5])[1]
    assert "must not decrease" in code([a, b], [0, 10, 5])[1]
    assert "overlap" in code([a, a], [0, 10, 20], fp=[0, 9])[1]
    assert "overlap" in code([a, a, a], [0, 10, 10, 12], fp=[0, 5, 6])[1]     # empty block between
    assert "aligned" in code([a], [0, 4], k=8)[1]
    with pytest.raises(kvlib.KVDecodeError):
        kvlib.kv_write_varlen(h, 1, 2, [a], [0, 4], 16, 16)                    # layers past the cache
    kvlib.kv_write_varlen(h, 0, 1, [], [0], None, None)                        # nothing to write
    kvlib.kv_cache_destroy(h)


def test_hand_worked_allocator_trace(kvlib):
    """The same trace as tests/golden/allocator_lazy_example.txt, through the library."""
    cfg = kvlib.make_config(1, 8, 8, 64, 8, 4, 4, page_size=16, flags=kvlib.KVC_FLAG_HOST_ONLY)
    # the library's page size is 16: scale the trace's page size 4 by 4
    h = kvlib.kv_cache_create(cfg)
    kvlib.kv_cache_set_page_order(h, [5, 2, 7, 0, 3, 6, 1, 4])
    a, b = kvlib.kv_seq_create(h), kvlib.kv_seq_create(h)
    assert (a, b) == (0, 1)
    kvlib.kv_seq_reserve(h, a, 17)     # positions 0..16: pages at 0 and 16
    kvlib.kv_seq_reserve(h, b, 16)
    kvlib.kv_begin_step(h, [a, b])     # a: position 17 (no page), b: position 16 (new page)
    assert kvlib.kv_seq_info(h, a) == (18, [5, 2])
    assert kvlib.kv_seq_info(h, b) == (17, [7, 0])
    kvlib.kv_seq_free(h, a)
    assert kvlib.kv_seq_create(h) == 0
    kvlib.kv_seq_reserve(h, 0, 33)
    assert kvlib.kv_seq_info(h, 0) == (33, [5, 2, 3])
    st = kvlib.kv_cache_query(h)
    assert st.free_pages == 3 and st.pages_in_use == 5 and st.live_seqs == 2
    kvlib.kv_cache_destroy(h)


def test_allocator_matches_oracle_model_on_random_traces(kvlib):
    P = 16
    for trial in range(4):
        rng = np.random.default_rng(100 + trial)
        num_pages, max_seqs, max_pages = 96, 12, 24
        cfg = kvlib.make_config(3, 28, 4, 128, num_pages, max_seqs, max_pages, flags=kvlib.KVC_FLAG_HOST_ONLY)
        h = kvlib.kv_cache_create(cfg)
        model = PagePoolModel(num_pages, P, max_seqs, max_pages)
        order = rng.permutation(num_pages)
        kvlib.kv_cache_set_page_order(h, order)
        model.set_page_order(order)
        live = []
        for it in range(400):
            r = rng.random()
            if r < 0.15:
                try:
                    s_model = model.seq_create()
                except OutOfPages:
                    with pytest.raises(kvlib.KVDecodeError) as ei:
                        kvlib.kv_seq_create(h)
                    assert ei.value.code == kvlib.KVC_ERR_OOM
                    continue
                assert kvlib.kv_seq_create(h) == s_model
                live.append(s_model)
            elif r < 0.25 and live:
                s = live.pop(int(rng.integers(len(live))))
                model.seq_free(s)
                kvlib.kv_seq_free(h, s)
            elif r < 0.6 and live:
                s = live[int(rng.integers(len(live)))]
                n = int(rng.integers(0, 70))
                try:
                    model.seq_reserve(s, n)
                    expect = None
                except OutOfPages:
                    expect = kvlib.KVC_ERR_OOM
                except ValueError:
                    expect = kvlib.KVC_ERR_INVALID
                if expect is None:
                    kvlib.kv_seq_reserve(h, s, n)
                else:
                    with pytest.raises(kvlib.KVDecodeError) as ei:
                        kvlib.kv_seq_reserve(h, s, n)
                    assert ei.value.code == expect
            elif live:
                k = int(rng.integers(1, len(live) + 1))
                batch = list(rng.choice(live, size=k, replace=False))
                try:
                    model.begin_step(batch)
                    expect = None
                except OutOfPages:
                    expect = kvlib.KVC_ERR_OOM
                except ValueError:
                    expect = kvlib.KVC_ERR_INVALID
                if expect is None:
                    kvlib.kv_begin_step(h, batch)
                else:
                    with pytest.raises(kvlib.KVDecodeError) as ei:
                        kvlib.kv_begin_step(h, batch)
                    assert ei.value.code == expect
            # bit-exact page tables and lengths
            for s in live:
                ln, pages = kvlib.kv_seq_info(h, s)
                assert ln == model.lens[s] and pages == model.pages[s], (trial, it, s)
            st = kvlib.kv_cache_query(h)
            assert st.pages_in_use == model.pages_in_use()
            assert st.free_pages == len(model.free)
            lens = [model.lens[s] for s in live]
            assert st.kv_bytes_allocated == oracle.kv_bytes_paged(3, 4, 128, P, lens)
        kvlib.kv_cache_destroy(h)


def test_begin_step_rejects_duplicates_and_dead_ids_without_changes(kvlib):
    h = host_cache(kvlib)
    a = kvlib.kv_seq_create(h)
    kvlib.kv_seq_reserve(h, a, 16)
    for bad in ([a, a], [a, 5], [-1]):
        with pytest.raises(kvlib.KVDecodeError) as ei:
            kvlib.kv_begin_step(h, bad)
        assert ei.value.code == kvlib.KVC_ERR_INVALID
    assert kvlib.kv_seq_info(h, a) == (16, kvlib.kv_seq_info(h, a)[1])
    assert kvlib.kv_seq_info(h, a)[0] == 16
    kvlib.kv_cache_destroy(h)


def test_begin_step_stops_at_a_full_page_row_without_changes(kvlib):
    """A row of max_pages pages takes positions up to max_pages * 16 - 1: the
    step that fills the last slot succeeds, the next one is refused and
    leaves the lengths and pages of every sequence in the batch as they were."""
    h = host_cache(kvlib, max_pages=4)
    a = kvlib.kv_seq_create(h)
    b = kvlib.kv_seq_create(h)
    kvlib.kv_seq_reserve(h, a, 63)
    kvlib.kv_seq_reserve(h, b, 10)
    kvlib.kv_begin_step(h, [a, b])
    assert kvlib.kv_seq_info(h, a)[0] == 64 and len(kvlib.kv_seq_info(h, a)[1]) == 4
    before = [kvlib.kv_seq_info(h, s) for s in (a, b)]
    free = kvlib.kv_cache_query(h).free_pages
    with pytest.raises(kvlib.KVDecodeError) as ei:
        kvlib.kv_begin_step(h, [b, a])
    assert ei.value.code == kvlib.KVC_ERR_INVALID
    assert [kvlib.kv_seq_info(h, s) for s in (a, b)] == before
    assert kvlib.kv_cache_query(h).free_pages == free
    kvlib.kv_cache_destroy(h)


def test_footprint_query_equals_eq1_when_lengths_fill_pages(kvlib):
    # LLaVA-7B shape: the worked example's 704 tokens are 44 whole pages
    cfg = kvlib.make_config(32, 32, 32, 128, 64, 2, 64, flags=kvlib.KVC_FLAG_HOST_ONLY)
    h = kvlib.kv_cache_create(cfg)
    s = kvlib.kv_seq_create(h)
    kvlib.kv_seq_reserve(h, s, 704)
    assert kvlib.kv_cache_query(h).kv_bytes_allocated == oracle.kv_bytes_eq1(32, 32, 128, 704) == 369_098_752
    kvlib.kv_cache_destroy(h)


def test_split_pages_range(kvlib):
    h = host_cache(kvlib)
    kvlib.kv_cache_set_split_pages(h, 0)
    kvlib.kv_cache_set_split_pages(h, 1024)
    with pytest.raises(kvlib.KVDecodeError):
        kvlib.kv_cache_set_split_pages(h, 1025)
    kvlib.kv_cache_destroy(h)


def test_noalloc_object_references_no_allocator(kvlib):
    """The entry point's translation unit calls no allocating routine: its
    object file (built from this repository's source) has no undefined
    reference to cudaMalloc*, cudaFree*, cuMemAlloc* or cuMemFree*."""
    import subprocess
    from paper_2603_12707_gb300 import _build
    obj = os.path.join(_build.OBJ, "kvd_noalloc.o")
    r = subprocess.run(["nm", "-u", "-C", obj], capture_output=True, text=True, check=True)
    bad = [l for l in r.stdout.splitlines()
           if any(s in l for s in ("cudaMalloc", "cudaFree", "cuMemAlloc", "cuMemFree", "cuMemCreate"))]
    assert not bad, bad
