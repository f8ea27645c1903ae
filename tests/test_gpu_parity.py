"""CUDA path against the CPU oracle, element by element, through the C ABI.

aq_pack and aq_decode must be bit-exact; aq_gemv must meet the product tolerance of
aq_testutil (relative Frobenius <= 2e-3, per element <= 1e-2*(1+|y_ref|)) against the oracle's
fp64 product. Sizes span several 32-row blocks and 32-group slices with ragged tails; the
full-size workloads are checked on sampled row ranges that include the last rows.
"""
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


RAGGED = [  # out, in, M, B, book dtype
    (1, 8, 1, 8, "f16"), (37, 560, 3, 8, "f16"), (100, 264, 4, 8, "bf16"),
    (33, 2056, 2, 8, "f16"), (50, 136, 2, 16, "f16"), (70, 520, 3, 16, "bf16"),
    (257, 1032, 4, 8, "f16"), (60, 1032, 8, 8, "f16"), (45, 264, 5, 8, "bf16"),
    (37, 560, 3, 4, "f16"), (100, 264, 4, 4, "bf16"),
    (40, 264, 8, 16, "f16"), (33, 520, 8, 4, "bf16"),
]


def _layer(out, inp, M, B, bd, seed):
    return workloads.make_layer(out, inp, G=8, M=M, B=B, book_dtype=bd, book_std=0.05,
                                scale_dtype=bd, seed=seed)


@pytest.mark.parametrize("case", RAGGED, ids=lambda c: "x".join(map(str, c)))
def test_pack_bit_exact(case):
    layer = _layer(*case, seed=17)
    lin = AQLinear.from_layer(layer)
    torch.cuda.synchronize()
    assert np.array_equal(lin.planes.cpu().numpy(), oracle.pack(layer))


@pytest.mark.parametrize("case", RAGGED, ids=lambda c: "x".join(map(str, c)))
def test_decode_bit_exact_ragged(case):
    layer = _layer(*case, seed=23)
    lin = AQLinear.from_layer(layer)
    for m in range(1, layer["M"] + 1):
        w = U.bits_of(lin.decode(m))
        assert np.array_equal(w, oracle.decode(layer, m)), m


@pytest.mark.parametrize("name", ["single_1024", "attn_4096"])
def test_decode_bit_exact_workloads(name):
    for _, layer in workloads.config_layers(name):
        lin = AQLinear.from_layer(layer)
        for m in range(1, layer["M"] + 1):
            got = U.bits_of(lin.decode(m))
            want = oracle.decode(layer, m)
            bad = np.flatnonzero(got != want)
            assert bad.size == 0, (m, bad[:8], got.ravel()[bad[:8]], want.ravel()[bad[:8]])


def test_decode_signed_zero_and_cancellation():
    """Planted +-0 codewords and exact cancellations: +0.0 start, fp32 order, one rounding."""
    layer = _layer(64, 512, 3, 8, "f16", seed=5)
    books = layer["books"].reshape(3, 256, 8).copy()
    books[0, :16] = 0x8000                       # -0.0
    books[1, :16] = 0x8000
    books[2, 16:32] = books[1, 16:32] ^ 0x8000   # exact negation of book 1 -> cancels to +0
    layer["books"] = books
    layer["codes"][:, :, :] = np.random.Generator(np.random.PCG64(1)).integers(
        0, 40, size=layer["codes"].shape, dtype=np.uint8)
    lin = AQLinear.from_layer(layer)
    for m in (1, 2, 3):
        assert np.array_equal(U.bits_of(lin.decode(m)), oracle.decode(layer, m)), m


def _gemv_check(layer, x_bits, x_dtype, m, y_dtype=None, rows=None, lin=None):
    lin = lin or AQLinear.from_layer(layer)
    x = x_to_device(x_bits, x_dtype)
    y = lin.gemv(x, m, y_dtype=y_dtype)
    y64 = U.to_f64(y)
    if rows is None:
        ref = oracle.product_exact(layer, x_bits, x_dtype, m)
        return U.assert_product_close(y64, ref, "m=%d" % m)
    errs = []
    for r0, r1 in rows:
        ref = oracle.product_exact(layer, x_bits, x_dtype, m, rows=(r0, r1))
        errs.append(U.assert_product_close(y64[:, r0:r1], ref, "m=%d rows %d:%d" % (m, r0, r1)))
    return errs


@pytest.mark.parametrize("case", RAGGED, ids=lambda c: "x".join(map(str, c)))
def test_gemv_ragged_every_batch(case):
    layer = _layer(*case, seed=29)
    lin = AQLinear.from_layer(layer)
    for batch in range(1, 17):
        x = workloads.make_x(batch, layer["in"], "f16", seed=batch)
        for m in range(1, layer["M"] + 1):
            _gemv_check(layer, x, "f16", m, lin=lin)


def test_gemv_single_1024():
    for _, layer in workloads.config_layers("single_1024"):
        x = workloads.config_x("single_1024", 1, layer["in"])
        for m in (1, 2):
            _gemv_check(layer, x, "f16", m)


@pytest.mark.parametrize("batch", [1, 4, 16])
def test_gemv_attn_4096(batch):
    (_, layer), = list(workloads.config_layers("attn_4096"))
    lin = AQLinear.from_layer(layer)
    x = workloads.config_x("attn_4096", batch, layer["in"])
    for m in (1, 2, 3, 4):
        _gemv_check(layer, x, "f16", m, lin=lin)


@pytest.mark.parametrize("batch", [1, 8])
def test_gemv_llama8b_block(batch):
    for lname, layer in workloads.config_layers("llama8b_block"):
        lin = AQLinear.from_layer(layer)
        x = workloads.config_x("llama8b_block", batch, layer["in"])
        out = layer["out"]
        rows = None if out <= 4096 else [(0, 1024), (out // 2, out // 2 + 512), (out - 1024, out)]
        for m in (1, 2, 3, 4):
            _gemv_check(layer, x, "bf16", m, rows=rows, lin=lin)


@pytest.mark.parametrize("batch", [1, 16])
def test_gemv_big_book_8192(batch):
    (_, layer), = list(workloads.config_layers("big_book_8192"))
    lin = AQLinear.from_layer(layer)
    x = workloads.config_x("big_book_8192", batch, layer["in"])
    for m in (1, 2):
        _gemv_check(layer, x, "f16", m, rows=[(0, 512), (4000, 4512), (8192 - 512, 8192)],
                    lin=lin)


@pytest.mark.parametrize("y_dtype", [aq.AQ_F32, aq.AQ_BF16, aq.AQ_F16])
def test_gemv_output_dtypes(y_dtype):
    layer = _layer(300, 1024, 2, 8, "f16", seed=3)
    x = workloads.make_x(1, 1024, "bf16", seed=2)
    for m in (1, 2):
        _gemv_check(layer, x, "bf16", m, y_dtype=y_dtype)
    x4 = workloads.make_x(4, 1024, "bf16", seed=2)
    _gemv_check(layer, x4, "bf16", 2, y_dtype=y_dtype)


def test_gemv_workspace_reuse_is_repeatable():
    """Counters are left at zero, so repeated calls on one workspace give identical bits."""
    layer = _layer(1000, 2048, 4, 8, "f16", seed=8)
    lin = AQLinear.from_layer(layer)
    x = x_to_device(workloads.make_x(1, 2048, "f16", seed=1), "f16")
    x3 = x_to_device(workloads.make_x(3, 2048, "f16", seed=1), "f16")
    for m in (1, 4):
        a = lin.gemv(x, m).clone()
        lin.gemv(x3, m)
        b = lin.gemv(x, m)
        assert torch.equal(a, b)


def test_gemv_prefix_buffer_only():
    """A buffer that holds only the first m planes is enough for a prefix-m call."""
    layer = _layer(200, 1024, 4, 8, "f16", seed=4)
    lin = AQLinear.from_layer(layer)
    x_bits = workloads.make_x(1, 1024, "f16", seed=9)
    x = x_to_device(x_bits, "f16")
    for m in (1, 2, 3):
        prefix = lin.planes_prefix(m).clone()
        ws = aq.workspace(aq.gemv_workspace_bytes(lin.layout, 1))
        y = torch.empty(1, 200, dtype=torch.float32, device="cuda")
        aq.aq_gemv(lin.layout, m, prefix, lin.books, lin.scales, x, aq.AQ_F16, 1, y, aq.AQ_F32, ws)
        U.assert_product_close(U.to_f64(y), oracle.product_exact(layer, x_bits, "f16", m))


def test_gemv_static_weights_flag_gives_same_result():
    """AQ_LAYOUT_STATIC_WEIGHTS only lets the kernel read the weights earlier; the result is
    bit-identical with and without it."""
    layer = _layer(2000, 4096, 4, 8, "f16", seed=12)
    lin = AQLinear.from_layer(layer)
    assert lin.layout.flags == aq.AQ_LAYOUT_STATIC_WEIGHTS
    for batch in (1, 3, 8):     # table lookups for 1 and 3 tokens, tensor cores for 8
        x = x_to_device(workloads.make_x(batch, 4096, "f16", seed=5), "f16")
        for m in (1, 3, 4):
            a = lin.gemv(x, m).clone()
            lin.layout.flags = 0
            b = lin.gemv(x, m).clone()
            lin.layout.flags = aq.AQ_LAYOUT_STATIC_WEIGHTS
            assert torch.equal(a, b), (batch, m)
