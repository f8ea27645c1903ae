"""Plant plausible mistakes in a copy of the oracle (on the CPU) and check that the pins catch
each one: a dropped scale, a wrong prefix bound, a transposed codebook, a reversed book order,
a sign error, wrong rounding, a wrong packing rotation, a wrong storage formula, and in the
distortion and loss a dropped normalisation, an off-by-one prefix, a sign error, a wrong
proxy Hessian power and shifted loss weights. A mutant that
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
    ("pack_4bit_nibble_order", "<< (4 * (p % 2))", "<< (4 * (1 - p % 2))"),
    ("reconstruct_drops_scale", "w_out[o * in + g * G + e] = s * acc;",
     "w_out[o * in + g * G + e] = acc;"),
]

# Mistakes planted in the Python part of the oracle (oracle/__init__.py): the distortion and
# loss of Sec. 2.2 / Sec. 5.
PY_MUTANTS = [
    ("wmse_drops_normalisation", "np.sum((E @ H) * E)) / out", "np.sum((E @ H) * E))"),
    ("wmse_prefix_off_by_one", "E = W - reconstruct_exact(layer, k)\n        res.append(float(np.sum((E @ H)",
     "E = W - reconstruct_exact(layer, max(1, k - 1))\n        res.append(float(np.sum((E @ H)"),
    ("wmse_sign_error", "E = W - reconstruct_exact(layer, k)\n        res.append(float(np.sum((E @ H)",
     "E = W + reconstruct_exact(layer, k)\n        res.append(float(np.sum((E @ H)"),
    ("wmse_squares_H", "np.sum((E @ H) * E)", "np.sum((E @ H @ H) * E)"),
    ("dbyd_shifted_weights", "total += lam[k] * D[k]", "total += lam[k] * D[k - 1]"),
    ("wmse_abs_keeps_sign_of_H", "A = np.abs(np.asarray(H, dtype=np.float64))",
     "A = np.asarray(H, dtype=np.float64)"),
    ("wmse_abs_drops_normalisation", "np.sum((E @ A) * E)) / out", "np.sum((E @ A) * E))"),
    ("beam_drops_cross_term", "h = [V[k][o, blk] - Sgg @ E[k][o, blk] for k in range(M)]",
     "h = [0.0 * V[k][o, blk] for k in range(M)]"),
    ("beam_uses_unsymmetrised_H", "    S = (H + H.T) / 2\n    lam = np.asarray(lam, dtype=np.float64)\n    E = [W - reconstruct_exact",
     "    S = H\n    lam = np.asarray(lam, dtype=np.float64)\n    E = [W - reconstruct_exact"),
    ("beam_weights_shifted", "score.append(sc + lam[t] * (q", "score.append(sc + lam[M - 1 - t] * (q"),
    ("beam_scale_dropped", "D = wg - s[o] * (P + books[t])", "D = wg - (P + books[t])"),
    ("beam_keeps_one_state", "keep = np.lexsort((cw, rank, score))[:K]",
     "keep = np.lexsort((cw, rank, score))[:1]"),
    ("wmse_abs_prefix_off_by_one", "E = np.abs(np.asarray(W, dtype=np.float64) - reconstruct_exact(layer, k))",
     "E = np.abs(np.asarray(W, dtype=np.float64) - reconstruct_exact(layer, max(1, k - 1)))"),
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


def _run_py_mutant(tmpdir, name, old, new):
    """A copy of the oracle package with one replacement in __init__.py, first on the path."""
    import shutil
    src_dir = os.path.join(ROOT, "oracle")
    pkg = os.path.join(tmpdir, name, "oracle")
    os.makedirs(pkg)
    for f in ("build.py", "oracle.cpp"):
        shutil.copy(os.path.join(src_dir, f), pkg)
    text = open(os.path.join(src_dir, "__init__.py")).read()
    assert old in text, "mutation site for %s not found in oracle/__init__.py" % name
    with open(os.path.join(pkg, "__init__.py"), "w") as f:
        f.write(text.replace(old, new))
    import oracle
    return (name,) + _run_pins(oracle.build.build(), first=os.path.join(tmpdir, name))


def _run_pins(lib, first=None):
    """Run every pin in a fresh interpreter against the oracle build `lib`: (exit code, output).
    Exit code 1 with a pin's name in the output means a pin failed."""
    path = ([first] if first else []) + [ROOT, os.path.join(ROOT, "tests")]
    env = dict(os.environ, ORACLE_LIB=lib, OMP_NUM_THREADS="1", PYTHONPATH=os.pathsep.join(path))
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
        futs += [ex.submit(_run_py_mutant, str(tmp_path), *m) for m in PY_MUTANTS]
        results = [f.result() for f in futs]
    survivors = [(n, out) for n, rc, out in results if rc == 0]
    assert not survivors, "mutants not caught by any pin: %s" % survivors
    # a caught mutant is one whose pins ran and at least one failed (not a crash on start-up)
    broken = [(n, out) for n, rc, out in results if "pin_" not in out]
    assert not broken, "mutant runs that did not reach the pins: %s" % broken
