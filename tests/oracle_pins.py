"""Pins of the CPU oracle to facts that do not come from the oracle itself.

Each pin_* function raises AssertionError when the oracle (the `oracle` package, possibly
loaded from another build via ORACLE_LIB) disagrees with:
  * a value the paper prints (App. C worked example of Eq. avg_bits),
  * an independent library routine (numpy float16 / torch bfloat16 rounding),
  * brute force in the paper's own notation (one-hot code vectors times C_m, Sec. 3.2 / Sec. 5),
  * exact rational arithmetic (fractions.Fraction) on dyadic inputs,
  * closed forms of special cases, or invariants (prefix linearity, prefix packing).
The same functions run under pytest (test_oracle_pins.py) and against deliberately broken
builds of the oracle (test_oracle_mutants.py), which must each fail at least one pin.
"""
import os
from fractions import Fraction

import numpy as np
import torch

import oracle
import workloads

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


# ---------------------------------------------------------------- storage model (App. C)

def pin_avg_bits_paper_example():
    """App. C: the 70B gate projection with g=8, M=2, B=8 costs approximately 2.002 bits."""
    with open(os.path.join(GOLDEN, "avg_bits_70b_gate_proj.txt")) as f:
        rows = [l.split() for l in f if l.strip() and not l.startswith("#")]
    for d_out, d_in, g, M, B, printed, decimals in rows:
        v = oracle.avg_bits(int(d_out), int(d_in), int(g), int(M), int(B))
        assert round(v, int(decimals)) == float(printed), (v, printed)


def pin_avg_bits_limit():
    """For huge layers the codebook and scale terms vanish: avg bits -> M*B/g (closed form)."""
    for (g, M, B) in [(8, 2, 8), (8, 4, 8), (8, 2, 16), (16, 3, 8)]:
        v = oracle.avg_bits(1 << 22, 1 << 22, g, M, B)
        assert abs(v - M * B / g) < 1e-3, (g, M, B, v)
        assert oracle.prefix_code_bits(g, M, B) == M * B / g


# ---------------------------------------------------------------- number formats

def _special_f32():
    vals = [0.0, -0.0, 1.0, -1.0, 65504.0, 65519.99, 65520.0, 1e6, -1e6, 6.1035156e-05,
            5.9604645e-08, 2.9802322e-08, 2.9802326e-08, 8.940697e-08, 1e-40, -1e-45,
            float("inf"), float("-inf"), 3.0e38, 3.4028235e38]
    # exact binary16 ties: midpoints between neighbouring fp16 values
    h = np.arange(0, 0x7c00, 97, dtype=np.uint16).view(np.float16).astype(np.float64)
    mids = (h[:-1] + np.nextafter(h[:-1].astype(np.float16), np.float16(np.inf)).astype(np.float64)) / 2
    return np.concatenate([np.array(vals, dtype=np.float64), mids, -mids]).astype(np.float32)


def pin_f16_rounding_matches_numpy():
    """float32 -> binary16 RNE against numpy's independent implementation."""
    rng = _rng(11)
    bits = rng.integers(0, 2**32, size=200000, dtype=np.uint64).astype(np.uint32)
    x = bits.view(np.float32)
    x = x[np.isfinite(x)]
    x = np.concatenate([x, _special_f32(), (rng.standard_normal(50000) * 1e-5).astype(np.float32)])
    got = oracle.round_bits(x, "f16")
    want = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(got, want), np.flatnonzero(got != want)[:10]


def pin_bf16_rounding_matches_torch():
    """float32 -> bfloat16 RNE against torch's independent implementation."""
    rng = _rng(12)
    bits = rng.integers(0, 2**32, size=200000, dtype=np.uint64).astype(np.uint32)
    x = bits.view(np.float32)
    x = x[np.isfinite(x)]
    ties = (rng.integers(0, 2**16, size=5000, dtype=np.uint32) << 16 | 0x8000).view(np.float32)
    x = np.concatenate([x, _special_f32(), ties[np.isfinite(ties)]])
    got = oracle.round_bits(x, "bf16")
    want = torch.from_numpy(x.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, want), np.flatnonzero(got != want)[:10]


def pin_widening_matches_numpy():
    """Every binary16 bit pattern widens to numpy's value (NaNs compared as NaN)."""
    allh = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    got = oracle.bits_value(allh, "f16")
    want = allh.view(np.float16).astype(np.float64)
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    assert same.all()
    b = np.arange(0, 1 << 16, 7, dtype=np.uint32).astype(np.uint16)
    got = oracle.bits_value(b, "bf16")
    want = torch.from_numpy(b.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    same = (got == want) | (np.isnan(got) & np.isnan(want))
    assert same.all()


# ---------------------------------------------------------------- reconstruction (Sec. 3.2, Sec. 5)

def _onehot_reconstruction(layer, m):
    """Brute force in the paper's notation: C_k is a g x 2^B matrix, b_{i,j,k} a one-hot
    vector in {0,1}^{2^B}; group j of row i is sum_{k<m} C_k b_{i,j,k}; the row is the
    concatenation of its groups; the scale multiplies the row (reading R1). fp64, exact."""
    out, inp, G, M, B = layer["out"], layer["in"], layer["G"], layer["M"], layer["B"]
    nb = 1 << B
    books = workloads_values(layer["books"], layer["book_dtype"]).reshape(M, nb, G)
    C = [books[k].T.copy() for k in range(M)]          # g x 2^B, column j = codeword j
    s = workloads_values(layer["scales"], layer["scale_dtype"])
    W = np.zeros((out, inp))
    for i in range(out):
        parts = []
        for j in range(inp // G):
            acc = np.zeros(G)
            for k in range(m):
                onehot = np.zeros(nb)
                onehot[int(layer["codes"][i, j, k])] = 1.0
                acc = acc + C[k] @ onehot
            parts.append(acc)
        W[i] = s[i] * np.concatenate(parts)
    return W


def workloads_values(bits, dtype):
    """Exact float64 values of bit patterns, via numpy / torch (not via the oracle)."""
    bits = np.asarray(bits, dtype=np.uint16)
    if dtype == "f16":
        return bits.view(np.float16).astype(np.float64)
    return torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).double().numpy()


def _tiny_layers():
    shapes = [(1, 8, 1, 8), (3, 16, 2, 8), (8, 24, 4, 8), (5, 8, 3, 16), (33, 40, 2, 8),
              (7, 24, 3, 4)]
    for idx, (out, inp, M, B) in enumerate(shapes):
        for bd in ("f16", "bf16"):
            yield workloads.make_layer(out, inp, G=8, M=M, B=B, book_dtype=bd, book_std=0.3,
                                       scale_dtype=bd, seed=100 + idx)


def pin_product_matches_onehot_bruteforce():
    """oracle_product_exact == x @ W^T with W from one-hot matrix products (fp64)."""
    for layer in _tiny_layers():
        x = workloads.make_x(3, layer["in"], "f16", seed=7)
        xv = x.view(np.float16).astype(np.float64)
        for m in range(1, layer["M"] + 1):
            W = _onehot_reconstruction(layer, m)
            want = xv @ W.T
            got = oracle.product_exact(layer, x, "f16", m)
            assert np.allclose(got, want, rtol=1e-12, atol=1e-12), (m, np.abs(got - want).max())


def pin_decode_matches_onehot_within_rounding():
    """oracle_decode == RNE(W) up to the fp32 summation error: at most one unit in the last
    place of the book format away from the exactly rounded one-hot reconstruction."""
    for layer in _tiny_layers():
        dt = layer["book_dtype"]
        for m in range(1, layer["M"] + 1):
            W = _onehot_reconstruction(layer, m)
            got = workloads_values(oracle.decode(layer, m), dt)
            if dt == "f16":
                ref = W.astype(np.float32).astype(np.float16).astype(np.float64)
                ulp = np.spacing(np.abs(ref).astype(np.float16)).astype(np.float64)
            else:
                ref = workloads_values(workloads.to_bits(W.astype(np.float32), "bf16"), "bf16")
                ulp = np.abs(ref) * 2.0 ** -7 + 2.0 ** -133
            assert np.all(np.abs(got - ref) <= ulp * 1.0001), (m, dt)


def pin_decode_exact_dyadic():
    """Dyadic inputs (multiples of 2^-10 in (-1,1), power-of-two scales): every fp32 step is
    exact, so decode must equal numpy's RNE of the exact one-hot reconstruction, bit for bit."""
    rng = _rng(5)
    for (out, inp, M) in [(7, 32, 4), (32, 64, 3)]:
        for dt in ("f16", "bf16"):
            layer = workloads.make_layer(out, inp, G=8, M=M, B=8, book_dtype=dt, scale_dtype=dt,
                                         seed=out)
            vals = rng.integers(-1023, 1024, size=layer["books"].shape) / 1024.0
            layer["books"] = workloads.to_bits(vals.astype(np.float32), dt)
            layer["scales"] = workloads.to_bits(
                2.0 ** rng.integers(-3, 4, size=out).astype(np.float32), dt)
            for m in range(1, M + 1):
                W = _onehot_reconstruction(layer, m)
                want = workloads.to_bits(W.astype(np.float32), dt)
                assert np.array_equal(oracle.decode(layer, m), want), (out, dt, m)


def pin_product_exact_rational():
    """Dyadic books, small-integer activations, unit scales: the fp64 product is exact, so it
    must equal the rational sum computed with Python Fractions."""
    rng = _rng(6)
    layer = workloads.make_layer(5, 24, G=8, M=3, B=8, book_dtype="f16", scale_dtype="f16", seed=9)
    vals = rng.integers(-1023, 1024, size=layer["books"].shape)
    layer["books"] = workloads.to_bits((vals / 1024.0).astype(np.float32), "f16")
    layer["scales"] = workloads.to_bits(np.ones(5, np.float32), "f16")
    xi = rng.integers(-8, 9, size=(2, 24))
    x = workloads.to_bits(xi.astype(np.float32), "f16")
    for m in (1, 2, 3):
        got = oracle.product_exact(layer, x, "f16", m)
        for t in range(2):
            for o in range(5):
                tot = Fraction(0)
                for g in range(3):
                    for e in range(8):
                        w = sum(Fraction(int(vals[k, layer["codes"][o, g, k], e]), 1024)
                                for k in range(m))
                        tot += Fraction(int(xi[t, g * 8 + e])) * w
                assert Fraction(got[t, o]) == tot, (m, t, o)


def pin_constant_codeword_closed_form():
    """All codes 0 and C_k[0] = constant vector c_k: y[t,o] = s[o]*(sum_k c_k)*sum_i x[t,i]."""
    rng = _rng(8)
    layer = workloads.make_layer(6, 32, G=8, M=4, B=8, seed=3)
    layer["codes"][:] = 0
    books = layer["books"].reshape(4, 256, 8).copy()
    c = workloads.to_bits(rng.standard_normal(4).astype(np.float32) * 0.1, "f16")
    books[:, 0, :] = c[:, None]
    layer["books"] = books
    x = workloads.make_x(2, 32, "f16", seed=4)
    xs = x.view(np.float16).astype(np.float64).sum(axis=1)
    s = layer["scales"].view(np.float16).astype(np.float64)
    cv = c.view(np.float16).astype(np.float64)
    for m in range(1, 5):
        want = np.outer(xs, s * cv[:m].sum())
        got = oracle.product_exact(layer, x, "f16", m)
        assert np.allclose(got, want, rtol=1e-12, atol=1e-13), m


def pin_onehot_codebook_selection():
    """One book whose codeword j is the unit vector e_(j mod 8): W is a scaled selection
    matrix, y[t,o] = s[o] * sum_g x[t, 8g + (b[o,g] mod 8)]."""
    layer = workloads.make_layer(9, 40, G=8, M=1, B=8, seed=12)
    books = np.zeros((1, 256, 8), np.float32)
    books[0, np.arange(256), np.arange(256) % 8] = 1.0
    layer["books"] = workloads.to_bits(books, "f16")
    x = workloads.make_x(3, 40, "f16", seed=5)
    xv = x.view(np.float16).astype(np.float64)
    s = layer["scales"].view(np.float16).astype(np.float64)
    got = oracle.product_exact(layer, x, "f16", 1)
    for t in range(3):
        for o in range(9):
            want = s[o] * sum(xv[t, 8 * g + int(layer["codes"][o, g, 0]) % 8] for g in range(5))
            assert abs(got[t, o] - want) <= 1e-12 * (1 + abs(want))


def pin_prefix_linearity():
    """Successive refinement (the nested increments of Sec. 4 / App. E): y_m - y_{m-1} equals
    the product with book m-1 alone (scaled by s), for every m."""
    for layer in _tiny_layers():
        x = workloads.make_x(2, layer["in"], "f16", seed=3)
        ys = [oracle.product_exact(layer, x, "f16", m) for m in range(1, layer["M"] + 1)]
        for m in range(2, layer["M"] + 1):
            single = dict(layer)
            single["M"] = 1
            nb = 1 << layer["B"]
            single["books"] = np.ascontiguousarray(
                layer["books"].reshape(layer["M"], nb, layer["G"])[m - 1])
            single["codes"] = np.ascontiguousarray(layer["codes"][:, :, m - 1:m])
            inc = oracle.product_exact(single, x, "f16", 1)
            scale = 1 + np.abs(ys[m - 1]).max()
            assert np.allclose(ys[m - 1] - ys[m - 2], inc, rtol=0, atol=1e-12 * scale), m


def pin_full_prefix_uses_every_book():
    """m = M reconstructs with all books: changing any single book changes y at m = M, and
    changing book M-1 leaves every m < M untouched."""
    layer = workloads.make_layer(4, 16, G=8, M=3, B=8, book_std=0.2, seed=21)
    x = workloads.make_x(1, 16, "f16", seed=2)
    base = [oracle.product_exact(layer, x, "f16", m) for m in (1, 2, 3)]
    for k in range(3):
        alt = dict(layer)
        books = layer["books"].reshape(3, 256, 8).copy()
        books[k] = workloads.to_bits(np.full((256, 8), 0.5, np.float32), "f16")
        alt["books"] = books
        ys = [oracle.product_exact(alt, x, "f16", m) for m in (1, 2, 3)]
        assert not np.allclose(ys[2], base[2])
        for m in range(1, 4):
            if m <= k:
                assert np.array_equal(ys[m - 1], base[m - 1]), (k, m)


def pin_dense_product_of_decode():
    """product_dense(decode) stays within the book-format rounding of product_exact."""
    layer = workloads.make_layer(16, 64, G=8, M=2, B=8, book_std=0.1, seed=31)
    x = workloads.make_x(2, 64, "f16", seed=8)
    for m in (1, 2):
        a = oracle.product_exact(layer, x, "f16", m)
        b = oracle.product_dense(oracle.decode(layer, m), "f16", x, "f16")
        bound = np.abs(x.view(np.float16).astype(np.float64)).sum(axis=1, keepdims=True) * 0.1 * 4 * 2.0 ** -10
        assert np.all(np.abs(a - b) <= bound + 1e-12), m


# ---------------------------------------------------------------- distortion (Sec. 2.2, Sec. 5)

def _wmse_case(out=24, inp=64, M=3, seed=7, dt="bf16"):
    """A layer, an 'original' weight W near its full reconstruction, and an activation matrix."""
    layer = workloads.make_layer(out, inp, G=8, M=M, B=8, book_dtype=dt, book_std=0.3,
                                 scale_dtype=dt, seed=seed)
    rng = _rng(seed + 1)
    W = _onehot_reconstruction(layer, M) + 0.05 * rng.standard_normal((out, inp))
    X = rng.standard_normal((inp, 2 * inp))
    return layer, W, X


def pin_reconstruct_exact_matches_onehot():
    """The exact W^(k) equals the one-hot brute force of Sec. 3.2 / Sec. 5 for every prefix."""
    for layer in _tiny_layers():
        for m in range(1, layer["M"] + 1):
            assert np.array_equal(oracle.reconstruct_exact(layer, m),
                                  _onehot_reconstruction(layer, m)), (layer["out"], m)


def pin_wmse_identity_is_frobenius():
    """X = I (H = I) reduces the weighted MSE to the plain MSE: D^(k) = ||W - W^(k)||_F^2 / d_out."""
    layer, W, _ = _wmse_case()
    D = oracle.wmse(layer, W, np.eye(layer["in"]))
    for k in range(1, layer["M"] + 1):
        E = W - _onehot_reconstruction(layer, k)
        want = sum(float(v) * float(v) for v in E.ravel()) / layer["out"]
        assert abs(D[k - 1] - want) <= 1e-12 * want, (k, D[k - 1], want)


def pin_wmse_trace_form_equals_activation_form():
    """The two sides of Eq. wmse-task: tr[E (X X^T / n) E^T] / d_out = ||E X||_F^2 / (d_out n)."""
    layer, W, X = _wmse_case()
    n = X.shape[1]
    D = oracle.wmse(layer, W, X @ X.T / n)
    for k in range(1, layer["M"] + 1):
        EX = (W - _onehot_reconstruction(layer, k)) @ X
        want = float(np.sum(EX * EX)) / (layer["out"] * n)
        assert abs(D[k - 1] - want) <= 1e-10 * want, (k, D[k - 1], want)


def pin_wmse_bruteforce_tiny():
    """Triple sum over rows and input pairs, in plain Python, on a 3 x 16 layer."""
    layer, W, X = _wmse_case(out=3, inp=16, M=2, seed=11, dt="f16")
    H = X @ X.T / X.shape[1]
    D = oracle.wmse(layer, W, H)
    for k in (1, 2):
        E = W - _onehot_reconstruction(layer, k)
        tot = 0.0
        for o in range(3):
            for i in range(16):
                for j in range(16):
                    tot += E[o, i] * H[i, j] * E[o, j]
        assert abs(D[k - 1] - tot / 3) <= 1e-10 * abs(tot / 3), (k, D[k - 1], tot / 3)


def pin_wmse_abs_bruteforce_tiny():
    """The magnitude behind the distortion tolerance, (1/d_out) sum_o |e_o| |H| |e_o|^T, as a
    triple sum over rows and input pairs in plain Python on a 3 x 16 layer."""
    layer, W, X = _wmse_case(out=3, inp=16, M=2, seed=17, dt="f16")
    H = X @ X.T / X.shape[1] - 0.3          # entries of both signs
    A = oracle.wmse_abs(layer, W, H)
    for k in (1, 2):
        E = W - _onehot_reconstruction(layer, k)
        tot = 0.0
        for o in range(3):
            for i in range(16):
                for j in range(16):
                    tot += abs(E[o, i]) * abs(H[i, j]) * abs(E[o, j])
        assert abs(A[k - 1] - tot / 3) <= 1e-10 * (tot / 3), (k, A[k - 1], tot / 3)


def pin_wmse_abs_equals_wmse_for_nonnegative_terms():
    """With W - W^(k) and H elementwise non-negative every term of the trace is non-negative,
    so the magnitude equals the distortion itself; in general it bounds |D^(k)| from above."""
    layer, _, X = _wmse_case(out=16, inp=48, M=3, seed=19, dt="f16")
    top = max(float(np.max(_onehot_reconstruction(layer, k))) for k in range(1, 4))
    rng = _rng(20)
    W = top + 0.01 + rng.random((16, 48))   # above every reconstruction: e >= 0
    H = np.abs(X @ X.T / X.shape[1])
    D, A = oracle.wmse(layer, W, H), oracle.wmse_abs(layer, W, H)
    assert np.all(np.abs(A - D) <= 1e-12 * A), (A, D)
    H2 = X @ X.T / X.shape[1] - 0.5
    W2 = _onehot_reconstruction(layer, 3) + 0.1 * rng.standard_normal((16, 48))
    D2, A2 = oracle.wmse(layer, W2, H2), oracle.wmse_abs(layer, W2, H2)
    assert np.all(np.abs(D2) <= A2 * (1 + 1e-12)) and np.any(np.abs(D2) < 0.9 * A2), (D2, A2)


def _beam_case(out, inp, M, B, seed):
    layer = workloads.make_layer(out, inp, G=8, M=M, B=B, book_std=0.3, seed=seed)
    rng = _rng(seed + 1)
    W = _onehot_reconstruction(layer, M) + 0.1 * rng.standard_normal((out, inp))
    X = rng.standard_normal((inp, 3 * inp))
    H = X @ X.T / X.shape[1] + 0.2 * rng.standard_normal((inp, inp))   # not symmetric
    return layer, W, H


def pin_beam_exhaustive_matches_bruteforce():
    """A beam wide enough to keep every partial state (K = (2^B)^(M-1)) returns, for every
    group, the code combination that minimises the row's Drop-by-Drop objective with the row's
    other groups held fixed; the objective is evaluated directly (full-row trace form, exact
    reconstruction) for all (2^B)^M combinations. Two weight matrices: one near a codeword
    combination, and one far from every combination, where a one-state (greedy) search picks a
    worse combination for some groups, so that the width of the beam is pinned too."""
    layer, W, H = _beam_case(6, 16, 2, 4, seed=41)
    W_far = _rng(45).standard_normal(W.shape) * 0.6
    lam = np.array([0.7, 0.3])
    greedy_differs = False
    for Wt in (W, W_far):
        got = oracle.beam_update(layer, Wt, H, lam, 16)
        greedy = oracle.beam_update(layer, Wt, H, lam, 1)
        for o in range(6):
            for g in range(2):
                best, arg = None, None
                for c0 in range(16):
                    for c1 in range(16):
                        trial = dict(layer)
                        trial["codes"] = layer["codes"].copy()
                        trial["codes"][o, g] = (c0, c1)
                        f = oracle.row_objective(trial, Wt, H, lam, o)
                        if best is None or f < best - 1e-12:
                            best, arg = f, (c0, c1)
                assert tuple(got[o, g]) == arg, (o, g, tuple(got[o, g]), arg)
                greedy_differs |= tuple(greedy[o, g]) != arg
    assert greedy_differs, "the case does not tell a beam from a greedy search"


def pin_beam_single_book_nearest_codeword():
    """One book, H = I, lambda = 1: the update is the nearest scaled codeword of each group,
    argmin_c ||w_g - s_o C[c]||^2, for any beam width."""
    layer, W, _ = _beam_case(4, 24, 1, 8, seed=43)
    books = workloads_values(layer["books"], "f16").reshape(256, 8)
    s = workloads_values(layer["scales"], "f16")
    for K in (1, 3):
        got = oracle.beam_update(layer, W, np.eye(24), [1.0], K)
        for o in range(4):
            for g in range(3):
                d = W[o, g * 8:(g + 1) * 8] - s[o] * books
                assert got[o, g, 0] == int(np.argmin(np.sum(d * d, axis=1))), (K, o, g)


def pin_wmse_vanishes_at_the_exact_weight():
    """W = W^(M): the full prefix has zero distortion; a shorter prefix leaves the dropped
    codebooks' contribution, which is positive for a positive definite H."""
    layer, _, X = _wmse_case(seed=13)
    M = layer["M"]
    W = _onehot_reconstruction(layer, M)
    D = oracle.wmse(layer, W, X @ X.T / X.shape[1])
    assert D[M - 1] == 0.0
    assert all(d > 0 for d in D[:-1]), D


def pin_wmse_invariances():
    """Only the symmetric part of H matters; D is linear in H; permuting rows (codes, scales
    and W together) changes nothing; the row sum splits over row blocks."""
    layer, W, X = _wmse_case(out=20, seed=17)
    rng = _rng(18)
    H = X @ X.T / X.shape[1]
    A = rng.standard_normal(H.shape)
    D = oracle.wmse(layer, W, H)
    assert np.allclose(oracle.wmse(layer, W, H + A - A.T), D, rtol=1e-12, atol=0)
    assert np.allclose(oracle.wmse(layer, W, 2.5 * H), 2.5 * D, rtol=1e-12, atol=0)
    perm = rng.permutation(layer["out"])
    pl = dict(layer, codes=np.ascontiguousarray(layer["codes"][perm]),
              scales=np.ascontiguousarray(layer["scales"][perm]))
    assert np.allclose(oracle.wmse(pl, W[perm], H), D, rtol=1e-12, atol=0)
    top = dict(layer, out=8, codes=np.ascontiguousarray(layer["codes"][:8]),
               scales=np.ascontiguousarray(layer["scales"][:8]))
    bot = dict(layer, out=12, codes=np.ascontiguousarray(layer["codes"][8:]),
               scales=np.ascontiguousarray(layer["scales"][8:]))
    split = (8 * oracle.wmse(top, W[:8], H) + 12 * oracle.wmse(bot, W[8:], H)) / 20
    assert np.allclose(split, D, rtol=1e-12, atol=0)


def _paper_loss_weights():
    out = {}
    with open(os.path.join(GOLDEN, "dbyd_loss_weights.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                name, *vals = line.split()
                out[name] = [float(Fraction(v)) for v in vals]
    return out


def pin_dbyd_loss_paper_weightings():
    """Sec. 5 / App. G.2 weightings: L = sum_k lambda_k D^(k) with lambda_k weighting prefix k.
    A unit distortion at prefix j alone gives lambda_j; Uni averages; 35W averages prefixes 3
    and 5; 345W averages prefixes 3, 4 and 5."""
    w = _paper_loss_weights()
    assert set(w) == {"Uni", "35W", "3W", "345W"}
    for name, lam in w.items():
        assert len(lam) == 5 and abs(sum(lam) - 1.0) < 1e-15, name
        for j in range(5):
            D = np.zeros(5)
            D[j] = 1.0
            assert oracle.dbyd_loss(D, lam) == lam[j], (name, j)
    D = np.array([16.0, 8.0, 4.0, 2.0, 1.0])
    assert abs(oracle.dbyd_loss(D, w["Uni"]) - 31.0 / 5) < 1e-14
    assert oracle.dbyd_loss(D, w["35W"]) == (4.0 + 1.0) / 2
    assert oracle.dbyd_loss(D, w["3W"]) == 4.0
    assert abs(oracle.dbyd_loss(D, w["345W"]) - 7.0 / 3) < 1e-15


# ---------------------------------------------------------------- packed planes

def pin_pack_positions():
    """Codes that spell their own coordinates: position p of row o in slice s must hold the
    code of group s*32 + (p+o) mod 32 of plane k; padding holds 0."""
    out, ng, M = 37, 70, 3
    inp = ng * 8
    codes = np.zeros((out, ng, M), np.uint16)
    for o in range(out):
        for g in range(ng):
            for k in range(M):
                codes[o, g, k] = 1 + g + 100 * k     # unique per (g, k), never 0
    layer = dict(out=out, **{"in": inp}, G=8, M=M, B=16, codes=codes)
    planes = oracle.pack(layer).view(np.uint16)
    rows_pad, ng_pad = 64, 96
    planes = planes.reshape(M, ng_pad // 32, rows_pad, 32)
    for k in range(M):
        for s in range(ng_pad // 32):
            for o in range(rows_pad):
                for p in range(32):
                    g = s * 32 + (p + o) % 32
                    want = (1 + g + 100 * k) if (o < out and g < ng) else 0
                    assert planes[k, s, o, p] == want


def pin_pack_positions_4bit():
    """4-bit codes: two per byte, position p of a (slice, row) unit in byte p // 2, low four
    bits for even p; the row rotation as for wider codes. Written out with plain loops."""
    out, inp, M = 37, 520, 3
    ng = inp // 8
    codes = np.zeros((out, ng, M), np.uint8)
    for o in range(out):
        for g in range(ng):
            for k in range(M):
                codes[o, g, k] = (3 * o + 5 * g + 7 * k) % 16
    layer = dict(out=out, **{"in": inp}, G=8, M=M, B=4, codes=codes)
    planes = oracle.pack(layer)
    rows_pad, ng_pad = 64, 96
    assert planes.size == M * rows_pad * ng_pad // 2
    planes = planes.reshape(M, ng_pad // 32, rows_pad, 16)
    for k in range(M):
        for s in range(ng_pad // 32):
            for o in range(rows_pad):
                for p in range(32):
                    g = s * 32 + (p + o) % 32
                    want = int(codes[o, g, k]) if (o < out and g < ng) else 0
                    byte = int(planes[k, s, o, p // 2])
                    got = (byte >> (4 * (p % 2))) & 15
                    assert got == want, (k, s, o, p)


def pin_pack_prefix_property():
    """The first m planes of a packed M-book layer equal the packed m-book truncation."""
    layer = workloads.make_layer(40, 272, G=8, M=4, B=8, seed=2)
    full = oracle.pack(layer)
    for m in (1, 2, 3):
        trunc = dict(layer)
        trunc["M"] = m
        trunc["codes"] = np.ascontiguousarray(layer["codes"][:, :, :m])
        p = oracle.pack(trunc)
        assert np.array_equal(full[: p.size], p), m


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]


if __name__ == "__main__":
    # Used by the mutation tests: run every pin, print the failing ones, exit 1 if any fail.
    import sys
    failed = []
    for fn in ALL_PINS:
        try:
            fn()
        except Exception as exc:  # noqa: BLE001 - any failure counts as a caught mutant
            failed.append("%s: %s" % (fn.__name__, type(exc).__name__))
    print("\n".join(failed) if failed else "all pins passed")
    sys.exit(1 if failed else 0)
