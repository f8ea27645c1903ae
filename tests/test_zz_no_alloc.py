"""The GEMV entry point that allocates nothing (aq_gemv_static_scratch), for callers that
cannot allocate device memory when they run a layer: its scratch comes from a fixed buffer
inside the library instead of a caller workspace. Called through the C ABI and compared with
aq_gemv (which takes a workspace) on two calls in a row, within the product tolerance used by
the other GEMV tests. This file is collected last on purpose."""
import ctypes

import pytest
import torch

import aq_testutil as U
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear, x_to_device

pytestmark = pytest.mark.gpu

CASES = [  # out, in, M, batch, x dtype
    (300, 1024, 3, 1, "f16"), (4096, 4096, 4, 1, "f16"), (257, 1032, 2, 5, "bf16"),
    (1024, 4096, 4, 16, "bf16"),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c)))
def test_static_scratch_matches_workspace_gemv(case):
    U.require_gpu()
    out, inp, M, batch, xd = case
    layer = workloads.make_layer(out, inp, G=8, M=M, B=8, book_std=0.05, seed=out + inp)
    lin = AQLinear.from_layer(layer)
    x = x_to_device(workloads.make_x(batch, inp, xd, seed=batch), xd)
    xc = aq.AQ_F16 if xd == "f16" else aq.AQ_BF16
    stream = torch.cuda.current_stream().cuda_stream
    for m in range(1, M + 1):
        ref = U.to_f64(lin.gemv(x, m, y_dtype=aq.AQ_F32))
        for _ in range(2):          # the shared buffer keeps the previous call's contents
            y = torch.full((batch, out), float("nan"), dtype=torch.float32, device="cuda")
            rc = aq.lib().aq_gemv_static_scratch(
                ctypes.byref(lin.layout), m, lin.planes.data_ptr(), lin.books.data_ptr(),
                lin.scales.data_ptr(), x.data_ptr(), xc, batch, y.data_ptr(), aq.AQ_F32, stream)
            assert rc == aq.AQ_OK, aq.status_string(rc)
            U.assert_product_close(U.to_f64(y), ref, "m=%d" % m)
    # no device-side wait gave up in any of these calls
    assert aq.lib().aq_gemv_static_scratch_status(stream) == aq.AQ_OK


def test_static_scratch_leaves_device_memory_alone():
    """A burst of calls changes the device's free memory by nothing: the entry point allocates
    neither memory of its own nor through the caching allocator (y is allocated up front)."""
    U.require_gpu()
    layer = workloads.make_layer(1000, 2048, G=8, M=3, B=8, book_std=0.05, seed=21)
    lin = AQLinear.from_layer(layer)
    x = x_to_device(workloads.make_x(1, 2048, "f16", seed=2), "f16")
    y = torch.empty(1, 1000, dtype=torch.float16, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream

    def call():
        rc = aq.lib().aq_gemv_static_scratch(
            ctypes.byref(lin.layout), 3, lin.planes.data_ptr(), lin.books.data_ptr(),
            lin.scales.data_ptr(), x.data_ptr(), aq.AQ_F16, 1, y.data_ptr(), aq.AQ_F16, stream)
        assert rc == aq.AQ_OK, aq.status_string(rc)

    call()                          # first call on the device: looks up the buffer's address
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(50):
        call()
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert aq.lib().aq_gemv_static_scratch_status(stream) == aq.AQ_OK


def test_static_scratch_rejects_sizes_beyond_the_buffer():
    U.require_gpu()
    L = aq.Layout.make(28672, 8192, 4)        # 32 slices x 16 tokens x 28672 rows of partials
    assert aq.gemv_workspace_bytes(L, 16) > (16 << 20)
    fake = 1 << 20
    rc = aq.lib().aq_gemv_static_scratch(ctypes.byref(L), 1, fake, fake, fake, fake, aq.AQ_F16,
                                         16, fake, aq.AQ_F16, None)
    assert rc == aq.AQ_ERR_WORKSPACE
