"""Prefill GEMM (tcgen05) against the CPU oracle through the C ABI.

Same product tolerance as the GEMV (relative Frobenius <= 2e-3, per element
<= 1e-2*(1+|y_ref|), against the oracle's fp64 product). Shapes cover several 512-token and
256-row pair tiles (including pairs whose second CTA has no rows), ragged token / row / input
tails, fp16 and bf16 books and activations, all
prefixes m <= 8 (five books, the paper's largest format, and more) and all output types; the 70B up-projection prefill is checked on sampled
token and row blocks that include the last ones.
"""
import ctypes

import numpy as np
import pytest
import torch

import aq_testutil as U
import oracle
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear, x_to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    U.require_gpu()


SHAPES = [  # tokens, out, in, M, dtype
    (1, 128, 64, 1, "f16"), (128, 128, 256, 2, "bf16"), (700, 300, 520, 3, "bf16"),
    (512, 256, 512, 4, "f16"), (1030, 260, 1032, 4, "bf16"), (37, 1000, 8, 2, "f16"),
    (600, 1288, 1032, 4, "bf16"), (700, 300, 520, 5, "bf16"), (256, 260, 1032, 8, "f16"),
    (1100, 256, 512, 6, "f16"),
]


@pytest.mark.parametrize("case", SHAPES, ids=lambda c: "x".join(map(str, c)))
@pytest.mark.parametrize("y_dtype", [aq.AQ_F32, aq.AQ_BF16, aq.AQ_F16])
def test_gemm_matches_oracle(case, y_dtype):
    tok, out, inp, M, dt = case
    layer = workloads.make_layer(out, inp, G=8, M=M, B=8, book_dtype=dt, book_std=0.05,
                                 scale_dtype=dt, seed=tok + out)
    lin = AQLinear.from_layer(layer)
    xb = workloads.make_x(tok, inp, dt, seed=7)
    x = x_to_device(xb, dt)
    for m in range(1, M + 1):
        y = lin.gemm(x, m, y_dtype=y_dtype)
        U.assert_product_close(U.to_f64(y), oracle.product_exact(layer, xb, dt, m), "m=%d" % m)


@pytest.mark.parametrize("case", [(2100, 300, 520, 5, "bf16"), (2048, 256, 1032, 3, "f16"),
                                  (2090, 1288, 520, 2, "bf16")],
                         ids=lambda c: "x".join(map(str, c)))
@pytest.mark.parametrize("y_dtype", [aq.AQ_F32, aq.AQ_BF16, aq.AQ_F16])
def test_gemm_dense_path_long_inputs(case, y_dtype):
    """From 2048 tokens, prefixes of two or more books decode W_m once into the workspace
    (fp16) and run TMA-fed pair MMAs on it: every prefix within the product tolerance. A
    16-bit y whose rows are a multiple of 16 bytes is written by bulk tensor stores from the
    operand rings (partial 32 x 32 chunks at a ragged row or token edge: 1288 rows, 2090
    tokens); 300 rows take the per-thread stores."""
    tok, out, inp, M, dt = case
    layer = workloads.make_layer(out, inp, G=8, M=M, B=8, book_dtype=dt, book_std=0.05,
                                 scale_dtype=dt, seed=tok + M)
    lin = AQLinear.from_layer(layer)
    xb = workloads.make_x(tok, inp, dt, seed=8)
    x = x_to_device(xb, dt)
    rows = np.r_[0:64, tok // 2:tok // 2 + 64, tok - 64:tok]
    for m in range(1, M + 1):
        y = lin.gemm(x, m, y_dtype=y_dtype)
        ys = U.to_f64(y[torch.as_tensor(rows, device="cuda")])
        U.assert_product_close(ys, oracle.product_exact(layer, xb[rows], dt, m), "m=%d" % m)


@pytest.mark.parametrize("tok,out,y_dtype", [(40, 300, aq.AQ_F32), (700, 300, aq.AQ_F32),
                                             (700, 296, aq.AQ_BF16)])
def test_gemm_4bit_codes(tok, out, y_dtype):
    """4-bit codes (16-entry codebooks): W_m decoded into the workspace, then the pair MMAs
    (with a bf16 y of 296 rows: the bulk-store epilogue)."""
    layer = workloads.make_layer(out, 520, G=8, M=4, B=4, book_dtype="bf16", book_std=0.05,
                                 scale_dtype="bf16", seed=tok)
    lin = AQLinear.from_layer(layer)
    xb = workloads.make_x(tok, 520, "bf16", seed=9)
    x = x_to_device(xb, "bf16")
    for m in range(1, 5):
        y = lin.gemm(x, m, y_dtype=y_dtype)
        U.assert_product_close(U.to_f64(y), oracle.product_exact(layer, xb, "bf16", m), "m=%d" % m)


def test_gemm_mixed_activation_and_book_types():
    """bf16 activations with fp16 books, and fp16 activations with bf16 books."""
    for bd, xd in (("f16", "bf16"), ("bf16", "f16")):
        layer = workloads.make_layer(200, 512, G=8, M=2, B=8, book_dtype=bd, book_std=0.05,
                                     scale_dtype=bd, seed=1)
        lin = AQLinear.from_layer(layer)
        xb = workloads.make_x(300, 512, xd, seed=2)
        for m in (1, 2):
            y = lin.gemm(x_to_device(xb, xd), m, y_dtype=aq.AQ_F32)
            U.assert_product_close(U.to_f64(y), oracle.product_exact(layer, xb, xd, m))


def test_gemm_agrees_with_gemv():
    layer = workloads.make_layer(384, 1024, G=8, M=4, B=8, book_std=0.05, seed=4)
    lin = AQLinear.from_layer(layer)
    x = x_to_device(workloads.make_x(16, 1024, "f16", seed=4), "f16")
    for m in (1, 4):
        a = U.to_f64(lin.gemm(x, m, y_dtype=aq.AQ_F32))
        b = U.to_f64(lin.gemv(x, m, y_dtype=aq.AQ_F32))
        U.assert_product_close(a, b)


def test_gemm_llama70b_up_prefill_sampled():
    (_, layer), = list(workloads.config_layers("llama70b_up_prefill"))
    lin = AQLinear.from_layer(layer)
    xb = workloads.config_x("llama70b_up_prefill", 4096, layer["in"])
    x = x_to_device(xb, "bf16")
    tok = np.r_[0:32, 2048:2064, 4064:4096]
    out = layer["out"]
    for m in (1, 2, 3, 4):
        y = lin.gemm(x, m, y_dtype=aq.AQ_F32)
        ys = U.to_f64(y[torch.as_tensor(tok, device="cuda")])
        for r0, r1 in ((0, 128), (out // 2, out // 2 + 128), (out - 128, out)):
            ref = oracle.product_exact(layer, xb[tok], "bf16", m, rows=(r0, r1))
            U.assert_product_close(ys[:, r0:r1], ref, "m=%d rows %d:%d" % (m, r0, r1))


def test_gemm_argument_errors():
    lib = aq.lib()
    fake = 1 << 20
    L = aq.Layout.make(256, 512, 4)
    ws_bytes = aq.gemm_workspace_bytes(L, 64)
    assert ws_bytes >= 256 + 64 * 512 * 2
    call = lambda L, m, tokens, wsb: lib.aq_gemm(ctypes.byref(L), m, fake, fake, fake, fake,
                                                 aq.AQ_BF16, tokens, fake, aq.AQ_F32, fake, wsb, None)
    assert call(L, 0, 64, ws_bytes) == aq.AQ_ERR_INVALID_ARG
    assert call(L, 1, -1, ws_bytes) == aq.AQ_ERR_INVALID_ARG
    assert call(L, 1, 64, ws_bytes - 16) == aq.AQ_ERR_WORKSPACE
    L16 = aq.Layout.make(256, 512, 2, B=16)
    assert call(L16, 1, 64, aq.gemm_workspace_bytes(L16, 64)) == aq.AQ_ERR_UNSUPPORTED
    assert call(L, 1, 0, 0) == aq.AQ_OK        # no tokens: nothing to do
