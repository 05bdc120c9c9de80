"""Mutation check of the oracle's pins.  Plausible mistakes are planted, one
at a time and on the CPU, in a copy of the oracle package (a dropped term, a
wrong sign or index, a transposed operand, a wrong layout stride, a changed
allocation policy); the pins of test_oracle_pins.py then run against the
copy, and every mutant must fail at least one of them.  Rewrites that cannot
change any result (for example another shift of the softmax maximum) are not
planted."""
import os
import shutil
import subprocess
import sys
import tempfile
from concurrent.futures import ThreadPoolExecutor

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (what the mistake is, file in oracle/, original text, planted text)
MUTANTS = [
    ("softmax scale dropped", "decode_oracle.c",
     "scores[t] = dot * scale;", "scores[t] = dot;"),
    ("sign of the max shift", "decode_oracle.c",
     "scores[t] = exp(scores[t] - mx);", "scores[t] = exp(mx - scores[t]);"),
    ("weights not normalised", "decode_oracle.c",
     "double w = scores[t] / z;", "double w = scores[t];"),
    ("GQA head mapping h % H_kv", "decode_oracle.c",
     "const int32_t g = h / G;", "const int32_t g = h % H_kv;"),
    ("K and V operands swapped", "decode_oracle.c",
     "k + base,\n                                    v + base,", "v + base,\n                                    k + base,"),
    ("dot product drops the last dim", "decode_oracle.c",
     "for (int32_t i = 0; i < d; ++i)\n            dot +=", "for (int32_t i = 0; i < d - 1; ++i)\n            dot +="),
    ("weighted sum reads the wrong element", "decode_oracle.c",
     "out[i] += w * bf16_bits_to_double(v[t * token_stride + i]);",
     "out[i] += w * bf16_bits_to_double(v[t * token_stride]);"),
    ("token stride ignores the KV heads", "decode_oracle.c",
     "n, (int64_t)H_kv * d, d, scale,", "n, (int64_t)d, d, scale,"),
    ("bf16 widening shifted by 15", "decode_oracle.c",
     "uint32_t w = ((uint32_t)bits) << 16;", "uint32_t w = ((uint32_t)bits) << 15;"),
    ("gather: slot from t / P", "decode_oracle.c",
     "const int64_t slot = t % P;\n        if (page < 0 || page >= num_pages) return -1;\n        for (int32_t g = 0; g < H_kv; ++g)\n            memcpy(dst",
     "const int64_t slot = t / P;\n        if (page < 0 || page >= num_pages) return -1;\n        for (int32_t g = 0; g < H_kv; ++g)\n            memcpy(dst"),
    ("scatter: page from t % P", "decode_oracle.c",
     "const int64_t page = page_table_row[t / P];\n        const int64_t slot = t % P;\n        if (page < 0 || page >= num_pages) return -1;\n        for (int32_t g = 0; g < H_kv; ++g)\n            memcpy(pool",
     "const int64_t page = page_table_row[t % P];\n        const int64_t slot = t % P;\n        if (page < 0 || page >= num_pages) return -1;\n        for (int32_t g = 0; g < H_kv; ++g)\n            memcpy(pool"),
    ("paged attention reads K from the V pool", "decode_oracle.c",
     "rc |= oracle_kv_gather(k_pool,", "rc |= oracle_kv_gather(v_pool,"),
    ("default scale 1/d", "__init__.py",
     "        scale = 1.0 / np.sqrt(d)\n    out = np.empty((B, H_q, d), dtype=np.float64)\n    ws =",
     "        scale = 1.0 / d\n    out = np.empty((B, H_q, d), dtype=np.float64)\n    ws ="),
    ("Eq. 1 without the factor 2 for K and V", "footprint.py",
     "return 2 * L * n_kv * d_h * s_ctx * b", "return L * n_kv * d_h * s_ctx * b"),
    ("paged footprint rounds down", "footprint.py",
     "P * ((int(n) + P - 1) // P)", "P * (int(n) // P)"),
    ("freed pages go to the back of the pop order", "allocator_model.py",
     "self.free = list(self.pages[seq]) + self.free", "self.free = self.free + list(self.pages[seq])"),
]


def _make_tree(tmp, mutant):
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(tmp, "oracle"),
                    ignore=shutil.ignore_patterns("*.so", "*.tmp*", "__pycache__"))
    os.makedirs(os.path.join(tmp, "tests"))
    for f in ("test_oracle_pins.py", "conftest.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), os.path.join(tmp, "tests", f))
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(tmp, "tests", "golden"))
    if mutant is not None:
        _, fname, old, new = mutant
        path = os.path.join(tmp, "oracle", fname)
        with open(path) as f:
            s = f.read()
        assert s.count(old) == 1, (fname, old)
        with open(path, "w") as f:
            f.write(s.replace(old, new))


def _pins_fail(mutant):
    """True if some pin fails against the oracle copy carrying `mutant`."""
    with tempfile.TemporaryDirectory() as tmp:
        _make_tree(tmp, mutant)
        env = {k: v for k, v in os.environ.items() if k != "PYTHONPATH"}
        env["OMP_NUM_THREADS"] = "2"
        r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                            os.path.join("tests", "test_oracle_pins.py")],
                           cwd=tmp, env=env, capture_output=True, text=True, timeout=900)
        return r.returncode != 0, r.stdout[-400:]


def test_unmutated_copy_passes_its_pins():
    failed, out = _pins_fail(None)
    assert not failed, out


def test_every_planted_mistake_fails_a_pin():
    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        results = list(ex.map(_pins_fail, MUTANTS))
    survivors = [m[0] for m, (failed, _) in zip(MUTANTS, results) if not failed]
    assert not survivors, f"mistakes no pin catches: {survivors}"
