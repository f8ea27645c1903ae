"""Failure detection without a GPU fault: a bounded device-side wait that nothing completes
gives up, records AQ_ERR_TIMEOUT in the workspace status word, and leaves the context usable
(the next call on the same stream runs and is checked against the oracle). The wait is the
same time-bounded mbarrier wait the compute kernels use (about 2 s)."""
import time

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


def test_bounded_wait_expires_and_the_context_survives():
    ws = aq.workspace(256)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    assert aq.lib().aq_selftest_wait(ws.data_ptr(), ws.numel(), None) == aq.AQ_OK
    assert aq.aq_workspace_status(ws) == aq.AQ_ERR_TIMEOUT      # synchronises the stream
    elapsed = time.perf_counter() - t0
    assert 1.0 < elapsed < 60.0, elapsed
    assert aq.aq_workspace_status(ws) == aq.AQ_OK               # reported once, then cleared
    layer = workloads.make_layer(64, 256, G=8, M=2, B=8, book_std=0.05, seed=3)
    lin = AQLinear.from_layer(layer)
    xb = workloads.make_x(1, 256, "f16", seed=4)
    y = lin.gemv(x_to_device(xb, "f16"), 2, y_dtype=aq.AQ_F32)
    U.assert_product_close(U.to_f64(y), oracle.product_exact(layer, xb, "f16", 2))
