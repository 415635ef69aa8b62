"""Each plausible mistake planted in a copy of the oracle is caught by a pin.

The mutants are built from the oracle's C source in a temporary directory and
run in child processes (a mutant may write out of bounds); the oracle itself
is never modified.
"""
import os
import subprocess
import sys

import pytest

import oracle

SRC = os.path.join(os.path.dirname(oracle.__file__), "kvs_oracle.c")
SRC_FP8 = os.path.join(os.path.dirname(oracle.__file__), "kvs_oracle_fp8.c")   # built beside it, unmutated
TESTS = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(TESTS)

MUTANTS = {
    "plane_order_swapped": ("int64_t p = 2 * l + kv;", "int64_t p = l + L * kv;"),
    "chunk_kv_swapped": ("((((l * 2 + kv) * n + i)", "((((l * 2 + (1 - kv)) * n + i)"),
    "chunk_layer_token_transposed": ("((((l * 2 + kv) * n + i) * H + h) * D) + d",
                                     "((((i * 2 + kv) * n + l) * H + h) * D) + d"),
    "paged_head_dim_transposed": ("return (slot * H + h) * D + d;", "return (slot * D + d) * H + h;"),
    "slot_offset_dropped": ("return phys * B + (t % B);", "return phys * B;"),
    "block_index_off_by_one": ("int64_t logical = t / B;", "int64_t logical = (t + 1) / B;"),
    "chunk_start_not_advanced": ("s += n;", "s += 0;"),
    "value_dropped": ("dropped_kv", None),
    "last_token_dropped": ("for (int64_t i = 0; i < n; ++i)", "for (int64_t i = 0; i + 1 < n; ++i)"),
    "store_reads_wrong_plane": ("else          chunk_el[b] = cache_el[b];",
                                "else          chunk_el[b] = (planes[p ^ 1] ? planes[p ^ 1] : plane)"
                                "[paged_elem(slot, h, d, H, D) * e + b];"),
}


def _mutate(name):
    src = open(SRC).read()
    old, new = MUTANTS[name]
    if name == "value_dropped":
        old, new = "for (int64_t kv = 0; kv < 2; ++kv)", "for (int64_t kv = 0; kv < 1; ++kv)"
    assert src.count(old) == 1, (name, src.count(old))
    return src.replace(old, new)


CHILD = r"""
import sys
sys.path[:0] = [{root!r}, {tests!r}]
import oracle, oracle_pins
lib = oracle.load({so!r})
failed = []
for pin in oracle_pins.ALL_PINS:
    try:
        pin(lib)
    except AssertionError as e:
        failed.append(pin.__name__)
print("FAILED:" + ",".join(failed))
"""


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(tmp_path, name):
    c = tmp_path / f"{name}.c"
    so = tmp_path / f"{name}.so"
    c.write_text(_mutate(name))
    subprocess.run(["gcc", "-O1", "-std=c11", "-shared", "-fPIC", str(c), SRC_FP8, "-o", str(so), "-lm"],
                   check=True)
    code = CHILD.format(root=ROOT, tests=TESTS, so=str(so))
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300)
    caught = r.returncode != 0 or ("FAILED:" in r.stdout and r.stdout.strip().split("FAILED:")[-1] != "")
    assert caught, f"mutant {name} passed every pin:\n{r.stdout}\n{r.stderr}"


def test_unmutated_copy_passes(tmp_path):
    """Control: the same harness on an unmodified copy reports no failure."""
    so = tmp_path / "clean.so"
    subprocess.run(["gcc", "-O1", "-std=c11", "-shared", "-fPIC", SRC, SRC_FP8, "-o", str(so), "-lm"], check=True)
    code = CHILD.format(root=ROOT, tests=TESTS, so=str(so))
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip().endswith("FAILED:"), r.stdout + r.stderr
