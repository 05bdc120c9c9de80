"""Pool slots that no sequence holds may contain anything: a page taken from
the free list keeps whatever its last owner (or a caller sharing the pool)
left there.  Every such slot, in every layer's K and V pools, is filled here
with NaN and Inf bit patterns before the steps run; the partial last page of
a row (and the page an append opens) then carries them in its rows past the
row's length.  The outputs must stay finite and match the float64 oracle,
which sees only the tokens each row holds, for MHA and every GQA group size
(2 to 8), head dims 64 and 128, fused and unfused launches, and item sizes
from one page up."""
import numpy as np
import pytest
import torch

from paper_2603_12707_gb300 import workloads as wl

from _gpu_common import Tracked, assert_close, bf16_to_f64, poison_unused_slots

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True, scope="module")
def _lib(kvlib):
    assert torch.cuda.is_available()
    yield


@pytest.mark.parametrize("split", [0, 1, 3])
@pytest.mark.parametrize("name,Hq,Hkv,d,lens", [
    ("mha128", 8, 8, 128, [1, 15, 16, 17, 33, 250]),
    ("gqa7_128", 28, 4, 128, [1, 14, 16, 31, 100, 257]),
    ("gqa3_128", 12, 4, 128, [2, 32, 47]),
    ("mha64", 8, 8, 64, [5, 16, 129]),
    ("gqa8_64", 16, 2, 64, [1, 15, 48, 99]),
    ("gqa2_64", 8, 4, 64, [3, 31, 64]),
    ("gqa4_128", 16, 4, 128, [9, 16, 70]),
    ("gqa5_128", 20, 4, 128, [1, 18, 45]),
    ("gqa6_64", 24, 4, 64, [7, 32, 81]),
    ("gqa8_128", 32, 4, 128, [2, 17, 150]),
])
def test_nan_and_inf_in_unheld_slots_never_reach_the_output(name, Hq, Hkv, d, lens, split):
    cfg = wl.custom(name, 2, Hq, Hkv, d, len(lens), lens=lens, seed=71 + Hq + d, page_order="shuffled")
    t = Tracked(cfg, extra_tokens=20, split_pages=split)
    assert poison_unused_slots(t.sess) > 0
    for step in range(3):
        t.begin_step()
        for layer in range(cfg.num_layers):
            out, q, _, _ = t.run_layer(layer, fused=(layer + step) % 2 == 0)
            torch.cuda.synchronize()
            got = bf16_to_f64(out)
            assert np.isfinite(got).all(), (name, split, step, layer)
            ref, vmax = t.oracle(layer, q)
            assert_close(got, ref, vmax, gqa=Hq > Hkv, what=(name, split, step, layer))
    t.close()
