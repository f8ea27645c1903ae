"""aq_beam_search against the CPU oracle: the code update of Alg. 1 ("update assignments b using
beam search", App. C), in the reading the oracle states (per group, a beam of width K over the
books in order, minimising the row's Drop-by-Drop objective with the other groups fixed).

Exact cases: codebook entries are multiples of 1/16 with |entry| <= 1/16, row scales 1 or 2,
weights multiples of 1/16 with |w| <= 1/4, H integer in [-1, 1] (so S = (H + H^T)/2 holds
halves) and lambda in {1, 2}. Then d = w_g - s (P + C_t[c]) is a multiple of 1/16 with
|d| <= 1.25 (eight books), every product and sum of the scores is a multiple of 1/512, and the
largest score (eight books, d_in <= 136) stays below 2^24 / 512: fp32 holds every score
exactly, both sides rank the candidates by the same numbers, ties included, and the codes must
be identical. Random cases (Gaussian weights, H = X X^T / n) compare on sampled groups: fp32
scores may order two candidates that tie to within rounding differently, so most groups must
match exactly and the others must reach the same objective to within rounding."""
import ctypes

import numpy as np
import pytest
import torch

import aq_testutil as U
import oracle
import oracle_pins
import paper_2606_12876_gb300 as aq
import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    U.require_gpu()


def _dt(name):
    return torch.float16 if name == "f16" else torch.bfloat16


def exact_case(out, inp, M, B, dt, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    nb = 1 << B
    books = rng.integers(-1, 2, size=(M, nb, 8)).astype(np.float32) / 16
    codes = rng.integers(0, nb, size=(out, inp // 8, M), dtype=np.uint8)
    scales = rng.choice(np.array([1.0, 2.0], np.float32), size=out)
    layer = dict(out=out, **{"in": inp}, G=8, M=M, B=B, books=workloads.to_bits(books, dt),
                 codes=codes, scales=workloads.to_bits(scales, dt), book_dtype=dt, scale_dtype=dt)
    W = rng.integers(-4, 5, size=(out, inp)).astype(np.float32) / 16
    H = rng.integers(-1, 2, size=(inp, inp)).astype(np.float32)
    return layer, workloads.to_bits(W, dt), H


def run_beam(layer, W_bits, H, lam, K, h_dtype=aq.AQ_F32, in_place=False):
    """aq_beam_search on device copies of the inputs; returns the new codes (numpy)."""
    dt = layer["book_dtype"]
    L = aq.Layout.make(layer["out"], layer["in"], layer["M"], B=layer["B"], book_dtype=dt,
                       scale_dtype=layer["scale_dtype"])
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    W = dev(W_bits.view(np.int16)).view(_dt(dt))
    codes = dev(layer["codes"])
    books = dev(layer["books"].view(np.int16))
    scales = dev(layer["scales"].view(np.int16))
    if h_dtype == aq.AQ_F32:
        h = dev(H.astype(np.float32))
    else:
        h = dev(workloads.to_bits(H.astype(np.float32), "bf16").view(np.int16))
    out = codes if in_place else torch.full_like(codes, 0xAB)
    ws = torch.empty(aq.beam_workspace_bytes(L), dtype=torch.uint8, device="cuda")
    aq.aq_beam_search(L, W, codes, books, scales, h, h_dtype, lam, K, out, ws)
    torch.cuda.synchronize()
    return out.cpu().numpy()


def W_values(W_bits, dt):
    return oracle_pins.workloads_values(W_bits, dt)


EXACT = [  # out, in, M, B, dtype, K, lambda, h dtype
    (37, 32, 2, 8, "f16", 1, None, aq.AQ_F32),
    (37, 32, 4, 8, "f16", 4, [1.0, 2.0, 1.0, 2.0], aq.AQ_F32),
    (21, 32, 3, 8, "bf16", 16, [2.0, 1.0, 1.0], aq.AQ_BF16),
    (45, 48, 3, 4, "f16", 16, None, aq.AQ_F32),
    (19, 32, 2, 4, "bf16", 16, [1.0, 2.0], aq.AQ_F32),      # K = 2^B: exhaustive
    (13, 32, 8, 8, "f16", 8, [2.0, 1.0, 2.0, 1.0, 1.0, 2.0, 1.0, 1.0], aq.AQ_F32),
    (70, 136, 2, 8, "f16", 6, [1.0, 1.0], aq.AQ_F32),        # d_in over three 64-wide tiles
]


@pytest.mark.parametrize("case", EXACT, ids=lambda c: "%dx%d_M%d_B%d_%s_K%d" % c[:6])
def test_beam_exact(case):
    out, inp, M, B, dt, K, lam, hdt = case
    layer, W_bits, H = exact_case(out, inp, M, B, dt, seed=out * 7 + inp + M)
    got = run_beam(layer, W_bits, H, lam, K, h_dtype=hdt)
    want = oracle.beam_update(layer, W_values(W_bits, dt), H.astype(np.float64),
                              lam if lam is not None else [1.0] * M, K)
    bad = np.argwhere(np.any(got != want, axis=2))
    assert bad.size == 0, "%d of %d groups differ, first (o, g) = %s: %s vs %s" % (
        len(bad), out * (inp // 8), tuple(bad[0]), got[tuple(bad[0])], want[tuple(bad[0])])


def test_beam_in_place():
    """codes_out == codes: the codes are read before any is written."""
    layer, W_bits, H = exact_case(29, 64, 3, 8, "f16", seed=3)
    got = run_beam(layer, W_bits, H, None, 4, in_place=True)
    want = oracle.beam_update(layer, W_values(W_bits, "f16"), H.astype(np.float64), [1.0] * 3, 4)
    assert np.array_equal(got, want)


def _rows(layer, rows):
    """The layer restricted to some rows (each row's search depends only on its own row)."""
    return dict(layer, out=len(rows), codes=np.ascontiguousarray(layer["codes"][rows]),
                scales=np.ascontiguousarray(layer["scales"][rows]))


def _group_objective(layer, W, H, lam, o, g, code_tuple):
    trial = dict(layer, codes=layer["codes"].copy())
    trial["codes"][o, g] = code_tuple
    return oracle.row_objective(trial, W, H, lam, o)


def _check_sampled(layer, W_bits, H, lam, K, got, rows, groups_per_row, seed):
    dt = layer["book_dtype"]
    rng = np.random.Generator(np.random.PCG64(seed))
    sub = _rows(layer, rows)
    W = W_values(W_bits, dt)[rows]
    ng = layer["in"] // 8
    pairs = [(i, int(g)) for i in range(len(rows))
             for g in rng.choice(ng, size=min(groups_per_row, ng), replace=False)]
    H64 = H.astype(np.float64)
    want = oracle.beam_update(sub, W, H64, lam, K, only=pairs)
    same = 0
    for i, g in pairs:
        a, b = tuple(got[rows[i], g]), tuple(want[i, g])
        if a == b:
            same += 1
            continue
        fa = _group_objective(sub, W, H64, lam, i, g, a)
        fb = _group_objective(sub, W, H64, lam, i, g, b)
        cur = _group_objective(sub, W, H64, lam, i, g, tuple(sub["codes"][i, g]))
        # the two searches took different branches at a near-tie: both ends must be as good
        # as each other to within the fp32 rounding of the scores
        assert fa <= fb + 1e-4 * abs(cur) + 1e-9, ("row", rows[i], "group", g, a, b, fa, fb)
    assert same >= 0.9 * len(pairs), "only %d of %d sampled groups match" % (same, len(pairs))


@pytest.mark.parametrize("out,inp,M,B,dt,K", [(300, 520, 4, 8, "f16", 8),
                                               (128, 1032, 2, 8, "bf16", 16),
                                               (96, 264, 3, 4, "f16", 4)])
def test_beam_random_sampled(out, inp, M, B, dt, K):
    """Gaussian weights near the current reconstruction, H = X X^T / n plus a small
    antisymmetric part (only S enters), lambda decreasing."""
    layer = workloads.make_layer(out, inp, G=8, M=M, B=B, book_dtype=dt, book_std=0.02,
                                 scale_dtype=dt, seed=out + inp)
    rng = np.random.Generator(np.random.PCG64(out))
    W = oracle.reconstruct_exact(layer, M) + 0.01 * rng.standard_normal((out, inp))
    W_bits = workloads.to_bits(W.astype(np.float32), dt)
    X = rng.standard_normal((inp, 2 * inp)).astype(np.float32)
    A = 0.05 * rng.standard_normal((inp, inp)).astype(np.float32)
    H = X @ X.T / X.shape[1] + (A - A.T)
    lam = [1.0 / (k + 1) for k in range(M)]
    got = run_beam(layer, W_bits, H, lam, K)
    rows = rng.choice(out, size=12, replace=False)
    _check_sampled(layer, W_bits, H, lam, K, got, rows, 6, seed=out + 1)


def test_beam_llama_attention_shape():
    """A 4096 x 4096 layer with four 2^8-entry books (the attention projection of the
    workloads), K = 8: sampled groups against the oracle."""
    out = inp = 4096
    M, K = 4, 8
    layer = workloads.make_layer(out, inp, G=8, M=M, B=8, seed=1)
    rng = np.random.Generator(np.random.PCG64(11))
    rows = np.sort(rng.choice(out, size=6, replace=False))
    W = oracle.reconstruct_exact(layer, M) + 0.01 * rng.standard_normal((out, inp))
    W_bits = workloads.to_bits(W.astype(np.float32), "f16")
    X = rng.standard_normal((inp, 256)).astype(np.float32)
    H = X @ X.T / 256 + 0.01 * np.eye(inp, dtype=np.float32)
    lam = [1.0, 0.5, 0.25, 0.125]
    got = run_beam(layer, W_bits, H, lam, K)
    assert got.shape == layer["codes"].shape
    _check_sampled(layer, W_bits, H, lam, K, got, rows, 4, seed=12)


def test_beam_zero_rows_is_a_no_op():
    L = aq.Layout.make(0, 64, 2)
    lib = aq.lib()
    assert lib.aq_beam_search(ctypes.byref(L), None, None, None, None, None, aq.AQ_F32, None, 4,
                              None, None, 0, None) == aq.AQ_OK
