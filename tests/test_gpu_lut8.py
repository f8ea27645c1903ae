"""The eight-token table-lookup GEMV (gemv_lut8: batch 5..8, prefixes up to six books, on
layers with at least 4560 (slice, book, 32-row block) items; y = x W_m^T of Sec. 2.2 with the
prefix reconstruction of Sec. 3.2 / Sec. 5). Its tables hold the tokens' products as fp16,
scaled per (token, slice, book) by a power of two, and four code bytes' entries are added in
fp16 before the fp32 sums, so these cases cover what the other GEMV tests do not reach at
small sizes: ragged rows and slices, every prefix it serves, mixed activation types,
activations of widely different magnitude per token, and exact arithmetic (where every fp16
entry and window sum is exact, the result must equal the oracle bit for bit)."""
import numpy as np
import pytest

import aq_testutil as U
import oracle
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear, x_to_device
from test_gpu_exact import assert_exact, exact_layer, exact_x

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    U.require_gpu()


def _check(layer, x_bits, xdt, m, batches):
    lin = AQLinear.from_layer(layer)
    x = x_to_device(x_bits, xdt)
    ref = oracle.product_exact(layer, x_bits, xdt, m)
    for b in batches:
        y = lin.gemv(x[:b], m, y_dtype=aq.AQ_F32)
        U.assert_product_close(U.to_f64(y), ref[:b], "m=%d batch=%d" % (m, b))


@pytest.mark.parametrize("bdt,xdt", [("f16", "f16"), ("f16", "bf16"), ("bf16", "bf16")])
def test_lut8_ragged(bdt, xdt):
    """1000 rows (ragged last row block), 8200 inputs (33 slices, the last with one group),
    six books: m = 3..6 take the eight-token kernel, m = 1, 2 the tensor-core kernel. Books are
    drawn as in the benchmark configurations, N(0, 0.02^2): with 11-bit table entries (as with
    the tf32 operands of the tensor-core kernel) the rounding error of one output grows like
    the square root of the number of (group, book) terms, and for this row length the
    per-element bound holds with margin only at that scale of weights."""
    layer = workloads.make_layer(1000, 8200, G=8, M=6, B=8, book_dtype=bdt, book_std=0.02,
                                 scale_dtype="f16", seed=11)
    x_bits = workloads.make_x(8, 8200, xdt, seed=12)
    for m in range(1, 7):
        _check(layer, x_bits, xdt, m, (5, 6, 7, 8))


def test_lut8_token_magnitudes():
    """Tokens whose activations differ by up to 10^8 in magnitude (bf16): each token's table
    is scaled on its own, so every token keeps fp16's relative precision. Checked with the
    relative Frobenius bound and, per element, the forward-error bound of the table form:
    each (group, book) entry is rounded once to fp16 and each pair of entries once more, so
    |y - y_exact| <= 2^-10 |s| sum_i |x_i| sum_k |C_k[b_k]_i| (the unit-scale bound
    1e-2 (1 + |y|) does not scale with the activations, and no 11-bit intermediate meets it
    where terms of order 1e4 cancel)."""
    rng = np.random.Generator(np.random.PCG64(5))
    layer = workloads.make_layer(640, 12288, G=8, M=4, B=8, book_dtype="bf16", book_std=0.3,
                                 scale_dtype="bf16", seed=6)
    x = rng.standard_normal((8, 12288)).astype(np.float32)
    x *= np.array([1e4, 1.0, 1e-4, 3e2, 2e-2, 7.0, 1e3, 5e-3], np.float32)[:, None]
    x[3, ::7] *= 50.0                                 # outliers inside one token
    x_bits = workloads.to_bits(x, "bf16")
    lin = AQLinear.from_layer(layer)
    xd = x_to_device(x_bits, "bf16")
    # |s| and |C_k| (sign bits cleared) give sum_k |C_k[b_k]| |s| per weight
    absl = dict(layer, books=np.asarray(layer["books"], np.uint16) & 0x7fff,
                scales=np.asarray(layer["scales"], np.uint16) & 0x7fff)
    X = np.abs((np.asarray(x_bits, np.uint16).astype(np.uint32) << 16).view(np.float32)).astype(np.float64)
    for m in (3, 4):
        ref = oracle.product_exact(layer, x_bits, "bf16", m)
        bound = 2.0 ** -10 * (X @ np.abs(oracle.reconstruct_exact(absl, m)).T)
        for b in (5, 8):
            y = U.to_f64(lin.gemv(xd[:b], m, y_dtype=aq.AQ_F32))
            rel = np.linalg.norm(y - ref[:b]) / np.linalg.norm(ref[:b])
            assert rel <= U.REL_FRO, "m=%d batch=%d: relative Frobenius error %.3e" % (m, b, rel)
            excess = np.abs(y - ref[:b]) - bound[:b]
            assert np.all(excess <= 0), "m=%d batch=%d: %d outputs beyond the bound, worst %.3e" % (
                m, b, int(np.sum(excess > 0)), float(excess.max()))


def test_lut8_exact():
    """Exact arithmetic (multiples of 1/16 in the books, power-of-two scales, integer
    activations): bit-identical to the oracle's fp64 product at batch 5..8."""
    layer = exact_layer(1000, 16384, 4, 8, "f16", seed=3)
    lin = AQLinear.from_layer(layer)
    x_bits = exact_x(8, 16384, "bf16", seed=4)
    x = x_to_device(x_bits, "bf16")
    for m in (3, 4):
        ref = oracle.product_exact(layer, x_bits, "bf16", m)
        for b in (5, 6, 7, 8):
            assert_exact(lin.gemv(x[:b], m, y_dtype=aq.AQ_F32), ref[:b], "m=%d batch=%d" % (m, b))


def test_lut8_refinement_chain_exact():
    """aq_gemv_refine at 8 tokens on a layer of 9216 rows x 4096 inputs: every step's one-book
    view has 16 x 288 = 4608 items, so each refinement runs the eight-token table kernel; the
    chain m = 1..4 (fp32, in place) equals each prefix product bit for bit."""
    layer = exact_layer(9216, 4096, 4, 8, "f16", seed=13)
    lin = AQLinear.from_layer(layer)
    x_bits = exact_x(8, 4096, "f16", seed=14)
    x = x_to_device(x_bits, "f16")
    y = None
    for m in range(1, 5):
        y = lin.refine(x, m, y, y=y)
        assert_exact(y, oracle.product_exact(layer, x_bits, "f16", m), "refine to m=%d" % m)
