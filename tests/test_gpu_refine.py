"""aq_gemv_refine against the CPU oracle: the increment x (s o C_{m-1}[b_{m-1}])^T that raises a
prefix-(m-1) product to prefix m (Sec. 4 successive reconstruction over the codebook prefixes of
Sec. 5). A chain of refinements from m = 1 must meet the product tolerance against the oracle's
prefix-m product at every step; the increment alone must match the oracle's y_m - y_(m-1);
in-place refinement must give the same bits as out-of-place."""
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


CASES = [  # out, in, M, B, dtype, batch (table lookups, tensor cores, direct, 16-bit codes)
    (300, 1032, 4, 8, "f16", 1), (257, 1032, 3, 8, "bf16", 3), (1000, 2048, 4, 8, "f16", 8),
    (60, 1032, 8, 8, "f16", 2), (96, 520, 2, 16, "f16", 1), (130, 264, 2, 16, "bf16", 5),
    (257, 1032, 4, 4, "f16", 1),
]


def _setup(case):
    out, inp, M, B, dt, batch = case
    layer = workloads.make_layer(out, inp, G=8, M=M, B=B, book_dtype=dt, book_std=0.05,
                                 scale_dtype=dt, seed=out + inp + M)
    xb = workloads.make_x(batch, inp, dt, seed=batch + 11)
    return layer, AQLinear.from_layer(layer), xb, x_to_device(xb, dt)


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c)))
def test_refinement_chain_matches_prefix_products(case):
    layer, lin, xb, x = _setup(case)
    y = None
    for m in range(1, layer["M"] + 1):
        y = lin.refine(x, m, y)             # fp32 result, y_prev = the prefix-(m-1) product
        ref = oracle.product_exact(layer, xb, case[4], m)
        U.assert_product_close(U.to_f64(y), ref, "m=%d" % m)


@pytest.mark.parametrize("case", CASES[:3], ids=lambda c: "x".join(map(str, c)))
def test_increment_alone_matches_oracle_difference(case):
    layer, lin, xb, x = _setup(case)
    prev = np.zeros((xb.shape[0], layer["out"]))
    for m in range(1, layer["M"] + 1):
        cur = oracle.product_exact(layer, xb, case[4], m)
        inc = lin.refine(x, m, None)
        U.assert_product_close(U.to_f64(inc), cur - prev, "increment m=%d" % m)
        prev = cur


def test_in_place_refinement_equals_out_of_place():
    layer, lin, xb, x = _setup(CASES[1])
    a = lin.refine(x, 1, None)
    b = a.clone()
    for m in range(2, layer["M"] + 1):
        a = lin.refine(x, m, a)                          # new buffer
        lin.refine(x, m, b, y=b)                         # in place
        assert torch.equal(a, b), m


def test_refinement_half_precision_output():
    """y_prev and y in fp16: each step rounds once; the chain stays near the prefix product."""
    layer, lin, xb, x = _setup(CASES[0])
    y = lin.refine(x, 1, None).half()
    for m in range(2, layer["M"] + 1):
        y = lin.refine(x, m, y)
        ref = oracle.product_exact(layer, xb, "f16", m)
        U.assert_product_close(U.to_f64(y), ref, "fp16 m=%d" % m)


def test_refine_argument_errors():
    layer, lin, xb, x = _setup(CASES[0])
    y = torch.empty(1, layer["out"], dtype=torch.float32, device="cuda")
    ws = aq.workspace(aq.gemv_workspace_bytes(lin.layout, 1))
    call = lambda m, y_prev: aq.lib().aq_gemv_refine(
        ctypes.byref(lin.layout), m, lin.planes.data_ptr(), lin.books.data_ptr(),
        lin.scales.data_ptr(), x.data_ptr(), aq.AQ_F16, 1, y_prev, y.data_ptr(), aq.AQ_F32,
        ws.data_ptr(), ws.numel(), None)
    assert call(0, None) == aq.AQ_ERR_INVALID_ARG
    assert call(layer["M"] + 1, None) == aq.AQ_ERR_INVALID_ARG
    assert call(1, y.data_ptr() + 4) == aq.AQ_ERR_ALIGNMENT
    assert call(2, y.data_ptr()) == aq.AQ_OK
    torch.cuda.synchronize()
