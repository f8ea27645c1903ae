"""Exact-arithmetic parity of the products on the GPU (Sec. 2.2 Y = W X with the prefix
reconstruction of Sec. 3.2 / Sec. 5).

The inputs are chosen so that every step of every kernel is exact: codebook entries are
multiples of 1/16 with |entry| <= 1/2 (a sum of up to eight of them has at most seven
significant bits, so it is exact in fp32 and, where a kernel rounds it to an MMA operand, in
fp16, bf16 and tf32), row scales are powers of two (0.5, 1, 2) and activations are integers in
[-3, 3]. Every table entry, partial sum and accumulator then holds a multiple of 1/32 below
2^18, which fp32 represents exactly, so any summation order gives the same value: the fp32
outputs must equal the oracle's fp64 product bit for bit. This pins what the tolerance-based
tests cannot: the reduction across slices and codebooks, where the scale enters, and that no
partial sum is dropped or counted twice."""
import numpy as np
import pytest
import torch

import aq_testutil as U
import oracle
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear, x_to_device

pytestmark = pytest.mark.gpu


def exact_layer(out, inp, M, B=8, book_dtype="f16", scale_dtype="f16", seed=0):
    rng = np.random.Generator(np.random.PCG64(seed))
    nb = 1 << B
    vals = rng.integers(-8, 9, size=(M, nb, 8)).astype(np.float32) / 16
    cdt = np.uint8 if B <= 8 else np.uint16
    codes = rng.integers(0, nb, size=(out, inp // 8, M), dtype=cdt)
    scales = rng.choice(np.array([0.5, 1.0, 2.0], np.float32), size=out)
    return dict(out=out, **{"in": inp}, G=8, M=M, B=B,
                books=workloads.to_bits(vals, book_dtype), codes=codes,
                scales=workloads.to_bits(scales, scale_dtype), book_dtype=book_dtype,
                scale_dtype=scale_dtype)


def exact_x(batch, inp, dtype, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    return workloads.to_bits(rng.integers(-3, 4, size=(batch, inp)).astype(np.float32), dtype)


def assert_exact(y, ref, what):
    y = U.to_f64(y)
    bad = np.argwhere(y != ref)
    assert bad.size == 0, "%s: %d of %d outputs differ, first at %s: %r vs %r" % (
        what, len(bad), y.size, tuple(bad[0]), y[tuple(bad[0])], ref[tuple(bad[0])])


# out, in, M, B, book dtype, x dtype: ragged rows and slices (in/8 not a multiple of 32),
# 8-bit codes with up to eight books, 4-bit and 16-bit codes, both activation types.
GEMV_CASES = [
    (300, 1032, 4, 8, "f16", "f16"),
    (97, 520, 8, 8, "bf16", "bf16"),
    (256, 2048, 3, 8, "f16", "bf16"),
    (130, 776, 4, 4, "f16", "f16"),
    (64, 264, 2, 16, "bf16", "f16"),
]


@pytest.mark.parametrize("case", GEMV_CASES, ids=lambda c: "x".join(map(str, c)))
def test_gemv_exact_every_batch(case):
    """aq_gemv at every batch 1..16 (every product kernel: table lookups, tensor-core tf32,
    4-bit tables, direct decode) with the shortest and the full prefix."""
    U.require_gpu()
    out, inp, M, B, bdt, xdt = case
    layer = exact_layer(out, inp, M, B, bdt, seed=out + inp)
    lin = AQLinear.from_layer(layer)
    x_bits = exact_x(16, inp, xdt, seed=inp)
    x = x_to_device(x_bits, xdt)
    for m in sorted({1, 2, M}):
        ref = oracle.product_exact(layer, x_bits, xdt, m)
        for batch in range(1, 17):
            y = lin.gemv(x[:batch], m, y_dtype=aq.AQ_F32)
            assert_exact(y, ref[:batch], "m=%d batch=%d" % (m, batch))


def test_gemv_refine_exact_chain():
    """A refinement chain m = 1..M (aq_gemv_refine, fp32, in place) equals each prefix
    product exactly."""
    U.require_gpu()
    layer = exact_layer(300, 1032, 4, seed=5)
    lin = AQLinear.from_layer(layer)
    x_bits = exact_x(3, 1032, "f16", seed=6)
    x = x_to_device(x_bits, "f16")
    for batch in (1, 3):
        y = None
        for m in range(1, 5):
            y = lin.refine(x[:batch], m, y, y=y)
            assert_exact(y, oracle.product_exact(layer, x_bits[:batch], "f16", m),
                         "refine to m=%d batch=%d" % (m, batch))


@pytest.mark.parametrize("case", [(200, 1032, 4, 8, "bf16", "bf16"), (96, 520, 8, 8, "f16", "f16"),
                                  (130, 776, 3, 4, "f16", "bf16")],
                         ids=lambda c: "x".join(map(str, c)))
def test_gemm_exact_both_forms(case):
    """aq_gemm with decoding in the loop (40 and 600 tokens) and, from 2048 tokens with two or
    more books (always for 4-bit codes), the form that decodes W_m once: exact outputs."""
    U.require_gpu()
    out, inp, M, B, bdt, xdt = case
    layer = exact_layer(out, inp, M, B, bdt, scale_dtype=bdt, seed=out * 3 + inp)
    lin = AQLinear.from_layer(layer)
    for tokens in (40, 600, 2048):
        x_bits = exact_x(tokens, inp, xdt, seed=tokens)
        x = x_to_device(x_bits, xdt)
        rows = np.r_[0:24, tokens - 24:tokens] if tokens > 48 else np.arange(tokens)
        for m in sorted({1, 2, M}):
            y = lin.gemm(x, m, y_dtype=aq.AQ_F32)[torch.as_tensor(rows, device=x.device)]
            assert_exact(y, oracle.product_exact(layer, x_bits[rows], xdt, m),
                         "tokens=%d m=%d" % (tokens, m))
