"""Plant plausible mistakes in a copy of the oracle (on the CPU) and check that the pins catch
each one: a dropped scale, a wrong prefix bound, a transposed codebook, a reversed book order,
a sign error, wrong rounding, a wrong packing rotation, a wrong storage formula. A mutant that
passes every pin would mean the pins could not tell that mistake from the truth."""
import concurrent.futures as cf
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.cpp")

MUTANTS = [
    ("decode_drops_scale", "const float v = acc * s;", "const float v = acc;"),
    ("product_drops_scale", "wrow[g * G + e] = s * acc;", "wrow[g * G + e] = acc;"),
    ("prefix_uses_all_books", "k < m; ++k", "k < M; ++k"),
    ("prefix_skips_first_book", "int k = 0; k < m", "int k = 1; k < m"),
    ("codebook_transposed", "(long)j * G + e]", "(long)e * (1L << B) + j]"),
    ("book_order_reversed", "(o * ng + g) * M + k)", "(o * ng + g) * M + (M - 1 - k))"),
    ("decode_sign_error", "acc = acc + bits_to_float", "acc = acc - bits_to_float"),
    ("f16_ties_round_up", "(rem == 0x1000u && (h & 1u))", "(rem == 0x1000u)"),
    ("bf16_truncates", "if (rem > 0x8000u || (rem == 0x8000u && (keep & 1u))) keep += 1;", ""),
    ("f16_subnormal_shift", "const int shift = -1 - e;", "const int shift = -e;"),
    ("f16_widen_exponent", "expo - 25);", "expo - 24);"),
    ("x_reversed_in_product", "sum += bits_to_double(x[t * in + i], x_dtype) * wrow[i];",
     "sum += bits_to_double(x[t * in + (in - 1 - i)], x_dtype) * wrow[i];"),
    ("pack_rotation_wrong", "((p + o) % 32)", "((p + 32 - o % 32) % 32)"),
    ("avg_bits_without_M", "(double)M * (double)d_out", "(double)d_out"),
]


def _run_mutant(tmpdir, name, old, new):
    src = open(SRC).read()
    assert old in src, "mutation site for %s not found in oracle.cpp" % name
    mut_src = os.path.join(tmpdir, name + ".cpp")
    with open(mut_src, "w") as f:
        f.write(src.replace(old, new))
    lib = os.path.join(tmpdir, name + ".so")
    subprocess.run(["g++", "-O1", "-std=c++17", "-ffp-contract=off", "-fopenmp", "-shared",
                    "-fPIC", mut_src, "-o", lib], check=True)
    return (name,) + _run_pins(lib)


def _run_pins(lib):
    """Run every pin in a fresh interpreter against the oracle build `lib`: (exit code, output).
    Exit code 1 with a pin's name in the output means a pin failed."""
    env = dict(os.environ, ORACLE_LIB=lib, OMP_NUM_THREADS="1",
               PYTHONPATH=os.pathsep.join([ROOT, os.path.join(ROOT, "tests")]))
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    return r.returncode, r.stdout[-2000:] + r.stderr[-2000:]


def test_unmutated_oracle_passes_the_pin_script():
    """Control: the script the mutants run passes on the real oracle, so a mutant's failure is
    a pin failing, not the script failing to start."""
    import oracle
    rc, out = _run_pins(oracle.build.build())
    assert rc == 0 and "all pins passed" in out, out


def test_every_planted_mistake_is_caught(tmp_path):
    with cf.ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 2)) as ex:
        futs = [ex.submit(_run_mutant, str(tmp_path), *m) for m in MUTANTS]
        results = [f.result() for f in futs]
    survivors = [(n, out) for n, rc, out in results if rc == 0]
    assert not survivors, "mutants not caught by any pin: %s" % survivors
    # a caught mutant is one whose pins ran and at least one failed (not a crash on start-up)
    broken = [(n, out) for n, rc, out in results if "pin_" not in out]
    assert not broken, "mutant runs that did not reach the pins: %s" % broken
