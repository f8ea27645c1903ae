"""Prefix stores (dynamic loading, Sec. 1 and Sec. 5): a layer whose device memory holds only the
first m codebooks, raised and lowered at run time from the packed layer in host memory.

Every product of a store-backed layer must equal, bit for bit, the same call on the layer that
holds all M codebooks (the kernels are the same and read the same bytes), and meet the product
tolerance against the oracle; decode must be bit-exact against the oracle. The device memory the
store holds must follow the resident prefix in whole 2 MiB granules."""
import ctypes

import numpy as np
import time

import pytest
import torch

import aq_testutil as U
import oracle
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear, x_to_device

pytestmark = pytest.mark.gpu

GRANULE = 2 << 20


@pytest.fixture(scope="module", autouse=True)
def gpu():
    U.require_gpu()


CASES = [  # out, in, M, B, dtype (planes of exactly one granule; small and ragged; 16-bit codes)
    (4096, 4096, 4, 8, "f16"), (300, 1032, 4, 8, "bf16"), (96, 520, 3, 16, "f16"),
    (200, 520, 4, 4, "bf16"),
]


def _setup(case, seed=0):
    out, inp, M, B, dt = case
    layer = workloads.make_layer(out, inp, G=8, M=M, B=B, book_dtype=dt, book_std=0.05,
                                 scale_dtype=dt, seed=out + inp + M + seed)
    full = AQLinear.from_layer(layer)
    return layer, full, full.to_host()


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c)))
def test_raise_and_lower_give_the_full_layers_results(case):
    layer, full, host = _setup(case)
    M, dt = case[2], case[4]
    xb = workloads.make_x(3, case[1], dt, seed=5)
    x = x_to_device(xb, dt)
    dyn = AQLinear.from_host(host, 1)
    try:
        for m in list(range(1, M + 1)) + [2, 1, M]:        # raise one by one, lower, re-raise
            dyn.set_prefix(m)
            for j in range(1, m + 1):
                assert torch.equal(dyn.gemv(x[:1], j), full.gemv(x[:1], j)), (m, j)
                assert torch.equal(dyn.gemv(x, j), full.gemv(x, j)), (m, j)
            assert np.array_equal(U.bits_of(dyn.decode(m)), oracle.decode(layer, m)), m
            U.assert_product_close(U.to_f64(dyn.gemv(x, m, y_dtype=aq.AQ_F32)),
                                   oracle.product_exact(layer, xb, dt, m), "m=%d" % m)
    finally:
        dyn.close()


def test_device_memory_follows_the_prefix():
    layer, full, host = _setup(CASES[0])
    pb = aq.plane_bytes(full.layout)
    assert pb == GRANULE                          # 4096 rows x 512 groups of 8-bit codes
    dyn = AQLinear.from_host(host, 1)
    try:
        head = dyn.device_bytes() - pb            # scales and all codebooks, one granule
        assert head == GRANULE
        for m in (2, 3, 4, 1, 0, 3):
            dyn.set_prefix(m)
            torch.cuda.current_stream().synchronize()   # a lowering's release follows its stream
            assert dyn.device_bytes() == head + m * pb, m
        with pytest.raises(ValueError):
            dyn.gemv(x_to_device(workloads.make_x(1, 4096, "f16", seed=1), "f16"), 4)
    finally:
        dyn.close()
    assert dyn.resident == 0


def test_lowering_does_not_wait_for_other_streams():
    """Lowering the prefix is ordered on the caller's stream only: a long kernel running on
    another stream does not hold the call up, and the dropped planes' memory is released once
    the caller's stream has passed the call. A raise straight after a lowering takes the
    dropped allocations back, and results stay those of the fully resident layer."""
    layer, full, host = _setup(CASES[0])
    pb = aq.plane_bytes(full.layout)
    dyn = AQLinear.from_host(host, 4)
    x = x_to_device(workloads.make_x(1, layer["in"], "f16", seed=5), "f16")
    try:
        head = dyn.device_bytes() - 4 * pb
        side = torch.cuda.Stream()
        torch.cuda.synchronize()
        with torch.cuda.stream(side):
            torch.cuda._sleep(400_000_000)          # a few hundred ms of spinning on `side`
        t0 = time.perf_counter()
        dyn.set_prefix(2)
        took = time.perf_counter() - t0
        still_running = not side.query()
        assert still_running and took < 0.05, (took, still_running)
        dyn.set_prefix(3)                           # straight back up: plane 2 is taken back
        torch.cuda.current_stream().synchronize()
        assert torch.equal(dyn.gemv(x, 3), full.gemv(x, 3))
        dyn.set_prefix(1)
        torch.cuda.current_stream().synchronize()
        assert dyn.device_bytes() == head + pb
        side.synchronize()
    finally:
        dyn.close()


def test_refinement_while_loading():
    """Load codebook m, then raise the result from prefix m-1 to m: the chain matches the
    full layer's refinement chain bit for bit and the oracle's prefix products."""
    case = CASES[1]
    layer, full, host = _setup(case)
    dt = case[4]
    xb = workloads.make_x(1, case[1], dt, seed=9)
    x = x_to_device(xb, dt)
    dyn = AQLinear.from_host(host, 1)
    try:
        y = dyn.refine(x, 1, None)
        y_full = full.refine(x, 1, None)
        for m in range(2, case[2] + 1):
            dyn.set_prefix(m)                     # copies on the current stream, then the call
            y = dyn.refine(x, m, y)
            y_full = full.refine(x, m, y_full)
            assert torch.equal(y, y_full), m
            U.assert_product_close(U.to_f64(y), oracle.product_exact(layer, xb, dt, m), "m=%d" % m)
    finally:
        dyn.close()


def test_gemm_from_a_store():
    case = CASES[1]
    layer, full, host = _setup(case)
    xb = workloads.make_x(300, case[1], case[4], seed=3)
    x = x_to_device(xb, case[4])
    dyn = AQLinear.from_host(host, 2)
    try:
        for m in (1, 2):
            assert torch.equal(dyn.gemm(x, m, y_dtype=aq.AQ_F32), full.gemm(x, m, y_dtype=aq.AQ_F32))
        dyn.set_prefix(4)
        y = dyn.gemm(x, 4, y_dtype=aq.AQ_F32)
        assert torch.equal(y, full.gemm(x, 4, y_dtype=aq.AQ_F32))
        rows = np.arange(0, 300, 7)
        U.assert_product_close(U.to_f64(y)[rows], oracle.product_exact(layer, xb[rows], case[4], 4),
                               "gemm m=4")
    finally:
        dyn.close()


def test_sources_in_device_memory_and_reload_from_empty():
    case = CASES[1]
    layer, full, host = _setup(case)
    xb = workloads.make_x(2, case[1], case[4], seed=4)
    x = x_to_device(xb, case[4])
    dev_src = dict(host, planes=full.planes, books=full.books, scales=full.scales)
    dyn = AQLinear.from_host(dev_src, 3)
    try:
        assert torch.equal(dyn.gemv(x, 3), full.gemv(x, 3))
        dyn.set_prefix(0)                          # everything dropped, scales re-copied below
        dyn.set_prefix(2)
        assert torch.equal(dyn.gemv(x, 2), full.gemv(x, 2))
    finally:
        dyn.close()


def test_store_argument_errors():
    layer, full, host = _setup(CASES[1])
    lib = aq.lib()
    s = aq.aq_store_create(full.layout)
    try:
        P, Bk, Sc = (host[k].data_ptr() for k in ("planes", "books", "scales"))
        assert lib.aq_store_prefix(s) == 0
        assert lib.aq_store_set_prefix(s, 5, P, Bk, Sc, None) == aq.AQ_ERR_INVALID_ARG
        assert lib.aq_store_set_prefix(s, -1, P, Bk, Sc, None) == aq.AQ_ERR_INVALID_ARG
        assert lib.aq_store_set_prefix(s, 1, None, Bk, Sc, None) == aq.AQ_ERR_INVALID_ARG
        assert lib.aq_store_set_prefix(s, 1, P, Bk, None, None) == aq.AQ_ERR_INVALID_ARG
        assert lib.aq_store_prefix(s) == 0
        assert lib.aq_store_set_prefix(s, 2, P, Bk, Sc, None) == aq.AQ_OK
        assert lib.aq_store_set_prefix(s, 3, P, Bk, None, None) == aq.AQ_OK   # scales resident
        assert lib.aq_store_set_prefix(s, 1, None, None, None, None) == aq.AQ_OK  # lowering
        assert lib.aq_store_prefix(s) == 1
        for fn in (lib.aq_store_planes, lib.aq_store_books, lib.aq_store_scales):
            assert fn(s) % 16 == 0
    finally:
        assert lib.aq_store_destroy(s) == aq.AQ_OK
    torch.cuda.synchronize()
