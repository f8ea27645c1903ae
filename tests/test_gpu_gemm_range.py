"""The prefill GEMM over the whole range of its inputs (Sec. 2.2 Y = W X on the prefix
reconstruction of Sec. 5): bf16 activations with outliers far beyond fp16's range, codebooks
whose summed entries exceed 65504 (bf16 and fp16 books), and bf16 codebooks so small that
their sums would fall into fp16's subnormal range. The tensor-core operands are fp16; the
power-of-two scalings of the activation rows and of the codebooks must keep every one of
these within the product tolerance of the oracle's fp64 product, in both forms of the GEMM
(decoding in the loop, and W_m decoded once from 2048 tokens)."""
import numpy as np
import pytest
import torch

import aq_testutil as U
import oracle
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear, x_to_device

pytestmark = pytest.mark.gpu


def _layer(out, inp, M, B, book_dtype, book_std, seed):
    return workloads.make_layer(out, inp, G=8, M=M, B=B, book_dtype=book_dtype,
                                book_std=book_std, scale_dtype=book_dtype, seed=seed)


def _x_with_outliers(tokens, inp, dtype, seed, big):
    """N(0, 1) activations with a few outlier channels and one outlier token scaled by `big`."""
    rng = np.random.Generator(np.random.PCG64(seed))
    x = rng.standard_normal((tokens, inp)).astype(np.float32)
    cols = rng.choice(inp, size=4, replace=False)
    x[:, cols] *= big
    x[tokens // 2] *= big
    return workloads.to_bits(x, dtype)


def workloads_values(bits, dtype):
    b = np.asarray(bits, dtype=np.uint16)
    if dtype == "f16":
        return b.view(np.float16).astype(np.float64)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _check(lin, layer, x_bits, xdt, tokens, m):
    """Relative Frobenius error <= 2e-3 as for every product, and per element the
    forward-error bound of a dot product whose weights are rounded to fp16 and summed in fp32,
    |y - y_exact| <= 2^-10 * sum_i |x_i| |w_i| (the rounding unit 2^-11 of fp16, twice, for
    the accumulation). This bound scales with the inputs; the bound 1e-2 * (1 + |y_exact|)
    used for unit-scale workloads does not, and no fp16-operand product meets it where terms
    of order 1e4 cancel to a small sum."""
    x = x_to_device(x_bits, xdt)
    rows = np.r_[0:16, tokens // 2 - 4:tokens // 2 + 4, tokens - 16:tokens] if tokens > 48 else np.arange(tokens)
    y = U.to_f64(lin.gemm(x, m, y_dtype=aq.AQ_F32)[torch.as_tensor(rows, device=x.device)])
    ref = oracle.product_exact(layer, x_bits[rows], xdt, m)
    what = "tokens=%d m=%d" % (tokens, m)
    assert np.all(np.isfinite(y)), what + ": non-finite output"
    rel = np.linalg.norm(y - ref) / np.linalg.norm(ref)
    assert rel <= U.REL_FRO, "%s: relative Frobenius error %.3e" % (what, rel)
    X = np.abs(workloads_values(x_bits[rows], xdt))
    W = np.abs(oracle.reconstruct_exact(layer, m))
    bound = 2.0 ** -10 * (X @ W.T)
    worst = np.max(np.abs(y - ref) / bound)
    assert worst <= 1.0, "%s: per-element error %.2f x the dot-product bound" % (what, worst)


@pytest.mark.parametrize("tokens", [40, 600, 2048])
def test_gemm_bf16_activation_outliers(tokens):
    """|x| up to about 4e6 (bf16), far beyond fp16's 65504."""
    U.require_gpu()
    layer = _layer(260, 1032, 4, 8, "bf16", 0.015, seed=tokens)
    lin = AQLinear.from_layer(layer)
    x_bits = _x_with_outliers(tokens, 1032, "bf16", seed=tokens + 1, big=1e6)
    assert np.max(np.abs(x_bits.view(np.int16).astype(np.int64) & 0x7fff)) > 0x4780  # > 65504
    for m in (1, 2, 4):
        _check(lin, layer, x_bits, "bf16", tokens, m)


@pytest.mark.parametrize("book_dtype,B", [("bf16", 8), ("f16", 8), ("bf16", 4)])
def test_gemm_codebook_sums_beyond_fp16(book_dtype, B):
    """Codebook entries of order 3e4: sums of two or more books exceed 65504."""
    U.require_gpu()
    layer = _layer(200, 520, 4, B, book_dtype, 3.0e4 if book_dtype == "bf16" else 1.2e4, seed=B)
    vals = workloads_values(layer["books"], book_dtype)
    assert np.all(np.isfinite(vals))
    if book_dtype == "f16":
        assert np.max(np.abs(vals)) < 65504
    # the unscaled sums of the four books (scales are at most 1.5) exceed fp16's range
    assert np.max(np.abs(oracle.reconstruct_exact(layer, 4))) > 1.5 * 65504
    lin = AQLinear.from_layer(layer)
    for tokens in (40, 2048):
        x_bits = workloads.make_x(tokens, 520, book_dtype, seed=tokens)
        for m in (1, 2, 4):
            _check(lin, layer, x_bits, book_dtype, tokens, m)


def test_gemm_tiny_bf16_codebooks():
    """Codebook entries of order 1e-7 (bf16): fp16 would hold their sums only as subnormals
    or zero; the scaled-up codebooks keep the full fp16 significand."""
    U.require_gpu()
    layer = _layer(200, 520, 3, 8, "bf16", 1.0e-7, seed=31)
    lin = AQLinear.from_layer(layer)
    for tokens in (40, 2048):
        x_bits = workloads.make_x(tokens, 520, "bf16", seed=tokens + 7)
        for m in (1, 3):
            _check(lin, layer, x_bits, "bf16", tokens, m)
