"""The pins are strong enough: each plausible mistake planted in a copy of the oracle (a dropped
term, a wrong index, a swapped operand) makes at least one pin fail.  The mistakes are planted
in temporary copies compiled on the CPU; the oracle itself is untouched."""
import os
import subprocess
import sys

import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))

# Runs every pin against one compiled mutant in a child process (a mutant that writes out of
# bounds may crash, which also counts as caught) and prints the pins that failed.
_RUNNER = r"""
import sys
sys.path[:0] = [sys.argv[1], sys.argv[2]]
import _pins, oracle
lib = oracle.load_variant(sys.argv[3])
failed = []
for pin in _pins.ALL_PINS:
    try:
        pin(lib=lib)
    except AssertionError:
        failed.append(pin.__name__)
print("FAILED:" + ",".join(failed))
"""

# (name, text in cfa_oracle.c, replacement)
MUTANTS = [
    ("rne_drops_lsb", "u + 0x7FFFu + lowest_kept_bit", "u + 0x7FFFu"),
    ("rne_truncates", "(u + 0x7FFFu + lowest_kept_bit) >> 16", "u >> 16"),
    ("rne_rounds_half_up", "u + 0x7FFFu + lowest_kept_bit", "u + 0x8000u"),
    ("rne_nan_passthrough", "return 0x7FC0u; /* any NaN */", "return (uint16_t)(u >> 16);"),
    ("rne_nan_test_wrong", "mantissa != 0u) return", "mantissa == 0u) return"),
    ("row_offset_dropped", "(uint64_t)e_row[t] * row_elems", "(uint64_t)e_row[t]"),
    ("row_is_first_dim", "d_shape[8 * j + d_ndim[j] - 1]", "d_shape[8 * j]"),
    ("base_uses_src_size", "base_elem * (uint64_t)es_d", "base_elem * (uint64_t)es_s"),
    ("big_endian_read", "x |= (uint64_t)p[k] << (8 * k)",
     "x |= (uint64_t)p[k] << (8 * (nbytes - 1 - k))"),
    ("src_stride_wrong", "read_le(src + src_i * (uint64_t)es_s, es_s)",
     "read_le(src + src_i * (uint64_t)es_d, es_s)"),
    ("dst_stride_wrong", "dst + i * (uint64_t)es_d", "dst + i * (uint64_t)es_s"),
    ("checksum_of_source", "ck += y;", "ck += x;"),
    ("checksum_misses_last", "ck += y;", "if (i + 1 < n) ck += y;"),
    ("cast_ignored", "const uint64_t y = converts ? orc_convert(conv, x) : x;",
     "const uint64_t y = x;"),
    ("oob_check_off_by_elem", "if (base_elem + n > d_numel)", "if (base_elem + n > d_numel + 1)"),
    ("cover_not_counted", "+= 1u;", "+= 0u;"),
    ("stride_ignored", "const uint64_t src_i = (i / C) * stride + (i % C);",
     "const uint64_t src_i = i;"),
    ("f16_truncates", "double m = nearbyint(ldexp(v, 10 - E));",
     "double m = floor(ldexp(v, 10 - E));"),
    ("f16_subnormal_scale", "const double m = nearbyint(ldexp(v, 24));",
     "const double m = nearbyint(ldexp(v, 23));"),
    ("f16_to_f32_bias", "ldexp(1024.0 + (double)m, (int)e - 25)",
     "ldexp(1024.0 + (double)m, (int)e - 24)"),
    ("f16_nan_drops_sign", "return sign | 0x7E00u;", "return 0x7E00u;"),
    ("bf16_to_f32_shift", "return (uint32_t)b << 16;", "return (uint32_t)b << 15;"),
    ("f16_to_bf16_skips_rounding", "return oracle_rne_bf16(oracle_f16_to_f32(h));",
     "return (uint16_t)(oracle_f16_to_f32(h) >> 16);"),
    ("stride_uses_row_length", "const uint64_t stride = given ? given : C;",
     "const uint64_t stride = C;"),
]


def _run_mutant(name, old, new, workdir):
    """Compiles one mutant and runs every pin against it in a child process; returns the pins
    that failed, or None if the mutant crashed the child (which also counts as caught)."""
    src = open(oracle.SOURCE_PATH).read()
    if src.count(old) != 1:
        return f"mutation site for {name} not unique"
    c = os.path.join(workdir, f"{name}.c")
    so = os.path.join(workdir, f"{name}.so")
    with open(c, "w") as f:
        f.write(src.replace(old, new))
    subprocess.run(["gcc", "-O1", "-std=c11", "-shared", "-fPIC", c, "-o", so, "-lm"],
                   check=True)
    root = os.path.dirname(HERE)
    r = subprocess.run([sys.executable, "-c", _RUNNER, HERE, root, so],
                       capture_output=True, text=True, timeout=600)
    if r.returncode != 0:
        return None
    line = [ln for ln in r.stdout.splitlines() if ln.startswith("FAILED:")][-1]
    return [x for x in line[len("FAILED:"):].split(",") if x]


@pytest.fixture(scope="module")
def mutant_results(tmp_path_factory):
    """All mutants compiled and checked concurrently, one child process each."""
    from concurrent.futures import ThreadPoolExecutor
    workdir = str(tmp_path_factory.mktemp("oracle_mutants"))
    workers = max(1, min(8, len(os.sched_getaffinity(0))))
    ex = ThreadPoolExecutor(workers)
    futs = {name: ex.submit(_run_mutant, name, old, new, workdir) for name, old, new in MUTANTS}
    yield futs
    ex.shutdown(wait=True)


@pytest.mark.parametrize("name", [m[0] for m in MUTANTS])
def test_pins_catch_mutant(name, mutant_results):
    failed = mutant_results[name].result()
    assert not isinstance(failed, str), failed
    assert failed is None or failed, f"no pin caught mutant {name}"
