"""Each plausible mistake planted in a copy of the fp8 oracle is caught by a pin.

The mutants are built from ``oracle/kvs_oracle_fp8.c`` in a temporary directory
(beside an unmodified copy of ``kvs_oracle.c``) and run in child processes; the
oracle itself is never modified.
"""
import os
import subprocess
import sys

import pytest

import oracle

HERE = os.path.dirname(oracle.__file__)
SRC = os.path.join(HERE, "kvs_oracle_fp8.c")
SRC_BF16 = os.path.join(HERE, "kvs_oracle.c")
TESTS = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(TESTS)

MUTANTS = {
    "scale_index_transposed": ("memcpy(&s, chunk + ((l * 2 + kv) * H + h) * 4, sizeof s);",
                               "memcpy(&s, chunk + ((l * H + h) * 2 + kv) * 4, sizeof s);"),
    "scale_block_skipped": ("const uint8_t *codes = chunks[j] + hdr;", "const uint8_t *codes = chunks[j];"),
    "codes_kv_swapped": ("return ((((l * 2 + kv) * n + i) * H + h) * D) + d;",
                         "return ((((l * 2 + (1 - kv)) * n + i) * H + h) * D) + d;"),
    "codes_head_dim_transposed": ("return ((((l * 2 + kv) * n + i) * H + h) * D) + d;",
                                  "return ((((l * 2 + kv) * n + i) * D + d) * H) + h;"),
    "ties_away_from_zero": ("else pick = (k % 2 == 0) ? k : k + 1;", "else pick = k + 1;"),
    "overflow_to_nan": ("if (k == 0x7E) return (uint8_t)(sign | 0x7E);",
                        "if (k == 0x7E) return (uint8_t)(a > 448.0 ? 0x7F : (sign | 0x7E));"),
    "subnormal_exponent_wrong": ("v = ldexp((double)m / 8.0, 1 - 7);", "v = ldexp((double)m / 8.0, 0 - 7);"),
    "bias_wrong": ("v = ldexp(1.0 + (double)m / 8.0, e - 7);", "v = ldexp(1.0 + (double)m / 8.0, e - 8);"),
    "bf16_truncates": ("if (rest < 0x8000u) r = down;", "if (rest < 0x10000u) r = down;"),
    "amax_counts_non_finite": ("if (isfinite(x) && fabsf(x) > amax) amax = fabsf(x);",
                               "if (!isnan(x) && fabsf(x) > amax) amax = fabsf(x);"),
    "scale_divisor_wrong": ("float scale = amax > 0.0f ? amax / 448.0f : 1.0f;",
                            "float scale = amax > 0.0f ? amax / 240.0f : 1.0f;"),
    "inverse_wrong": ("float inv = amax > 0.0f ? 448.0f / amax : 1.0f;",
                      "float inv = amax > 0.0f ? 447.0f / amax : 1.0f;"),
    "store_uses_scale_not_inverse": ("float q = x * inv;", "float q = x * scale;"),
    "store_divides_by_inverse": ("float q = x * inv;", "float q = x / inv;"),
    "retrieve_ignores_scale": ("float y = x * scale;", "float y = x;"),
    "negative_zero_lost": ("uint8_t sign = signbit(v) ? 0x80 : 0x00;", "uint8_t sign = v < 0 ? 0x80 : 0x00;"),
}


def _mutate(name):
    src = open(SRC).read()
    old, new = MUTANTS[name]
    assert src.count(old) == 1, (name, src.count(old))
    return src.replace(old, new)


CHILD = r"""
import sys
sys.path[:0] = [{root!r}, {tests!r}]
import oracle, oracle_pins_fp8
lib = oracle.load({so!r})
failed = []
for pin in oracle_pins_fp8.ALL_PINS:
    try:
        pin(lib)
    except AssertionError as e:
        failed.append(pin.__name__)
print("FAILED:" + ",".join(failed))
"""


def _build_and_run(tmp_path, name, src_text):
    c = tmp_path / f"{name}.c"
    so = tmp_path / f"{name}.so"
    c.write_text(src_text)
    subprocess.run(["gcc", "-O1", "-std=c11", "-ffp-contract=off", "-shared", "-fPIC", str(c), SRC_BF16,
                    "-o", str(so), "-lm"], check=True)
    code = CHILD.format(root=ROOT, tests=TESTS, so=str(so))
    return subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=600)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_fp8_mutant_is_caught(tmp_path, name):
    r = _build_and_run(tmp_path, name, _mutate(name))
    caught = r.returncode != 0 or ("FAILED:" in r.stdout and r.stdout.strip().split("FAILED:")[-1] != "")
    assert caught, f"mutant {name} passed every pin:\n{r.stdout}\n{r.stderr}"


def test_unmutated_fp8_copy_passes(tmp_path):
    """Control: the same harness on an unmodified copy reports no failure."""
    r = _build_and_run(tmp_path, "clean", open(SRC).read())
    assert r.returncode == 0 and r.stdout.strip().endswith("FAILED:"), r.stdout + r.stderr
