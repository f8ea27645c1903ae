"""aq_wmse against the CPU oracle: the weighted MSE of Sec. 2.2 (Eq. wmse-task) of every prefix
of a packed layer, as Drop-by-Drop measures it (Sec. 5), and the Drop-by-Drop objective.

Tolerance (derived from the arithmetic): the GPU rounds E_k = W - W^(k) to bf16 twice (the MMA
operand and the epilogue copy) and the folded H once, each a relative error of at most
u = 2^-8, and accumulates in fp32. To first order |D - D_exact| <= (3u + fp32 terms) * D_abs
with D_abs = (1/d_out) sum_o |e_o||H||e_o|^T; the test allows 1.25e-2 * D_abs. The roundings
are unbiased and independent, so on these random inputs the error relative to D itself is far
below that bound: the test also requires |D - D_exact| <= 2e-3 * D_exact."""
import ctypes

import numpy as np
import pytest
import torch

import aq_testutil as U
import oracle
import oracle_pins
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear

pytestmark = pytest.mark.gpu

BOUND_ABS = 1.25e-2
BOUND_REL = 2e-3


@pytest.fixture(scope="module", autouse=True)
def gpu():
    U.require_gpu()


def _case(out, inp, M, dt, seed, noise=0.01, n_mult=2, B=8):
    """A layer, an 'original' weight W near its full reconstruction (rounded to the book type)
    and H = X X^T / n for Gaussian X (n = n_mult * in), as float32."""
    layer = workloads.make_layer(out, inp, G=8, M=M, B=B, book_dtype=dt, book_std=0.02,
                                 scale_dtype=dt, seed=seed)
    rng = np.random.Generator(np.random.PCG64(seed + 1))
    W = oracle.reconstruct_exact(layer, M) + noise * rng.standard_normal((out, inp))
    W_bits = workloads.to_bits(W.astype(np.float32), dt)
    X = rng.standard_normal((inp, n_mult * inp)).astype(np.float32)
    H = (X.astype(np.float64) @ X.T.astype(np.float64) / X.shape[1]).astype(np.float32)
    return layer, W_bits, H


def _device(layer, W_bits, H):
    lin = AQLinear.from_layer(layer)
    dt = torch.float16 if layer["book_dtype"] == "f16" else torch.bfloat16
    W = torch.from_numpy(W_bits.view(np.int16)).cuda().view(dt)
    return lin, W, torch.from_numpy(H).cuda()


def _check(layer, W_bits, H, d_gpu, what=""):
    W = oracle_pins.workloads_values(W_bits, layer["book_dtype"])
    ref = oracle.wmse(layer, W, H.astype(np.float64))
    absb = oracle.wmse_abs(layer, W, H.astype(np.float64))
    for k in range(layer["M"]):
        err = abs(d_gpu[k] - ref[k])
        assert err <= BOUND_ABS * absb[k], (what, k + 1, d_gpu[k], ref[k], absb[k])
        assert err <= BOUND_REL * ref[k], (what, k + 1, d_gpu[k], ref[k], err / ref[k])
    return ref


CASES = [  # out, in, M, dtype: several tiles; ragged rows and inputs; second pass; eight books
    (256, 512, 4, "bf16"), (300, 1032, 4, "f16"), (130, 264, 5, "bf16"), (64, 256, 8, "f16"),
    (1000, 2048, 2, "bf16"), (96, 64, 1, "f16"),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c)))
def test_wmse_matches_oracle(case):
    out, inp, M, dt = case
    layer, W_bits, H = _case(out, inp, M, dt, seed=out + inp + M)
    lin, W, Hd = _device(layer, W_bits, H)
    d = lin.wmse(W, Hd).cpu().numpy()
    ref = _check(layer, W_bits, H, d, str(case))
    if M > 1:
        assert all(ref[k] > ref[k + 1] for k in range(M - 1)), ref   # the fixture refines


def test_sixteen_bit_codes():
    layer, W_bits, H = _case(160, 520, 2, "bf16", seed=8, B=16)
    lin, W, Hd = _device(layer, W_bits, H)
    _check(layer, W_bits, H, lin.wmse(W, Hd).cpu().numpy(), "B=16")


def test_four_bit_codes():
    layer, W_bits, H = _case(130, 264, 4, "f16", seed=12, B=4)
    lin, W, Hd = _device(layer, W_bits, H)
    _check(layer, W_bits, H, lin.wmse(W, Hd).cpu().numpy(), "B=4")


def test_bf16_h_and_nonsymmetric_h():
    """H given in bf16, and a non-symmetric H (only its symmetric part counts)."""
    layer, W_bits, H = _case(200, 520, 3, "bf16", seed=3)
    rng = np.random.Generator(np.random.PCG64(4))
    A = (0.1 * rng.standard_normal(H.shape)).astype(np.float32)
    Hn = (H + A - A.T).astype(np.float32)
    lin, W, Hd = _device(layer, W_bits, Hn)
    _check(layer, W_bits, Hn, lin.wmse(W, Hd).cpu().numpy(), "non-symmetric")
    Hb = torch.from_numpy(H).cuda().to(torch.bfloat16)
    Hb64 = Hb.float().cpu().numpy()                       # the values the kernel is given
    _check(layer, W_bits, Hb64, lin.wmse(W, Hb).cpu().numpy(), "bf16 H")


def test_dbyd_loss_with_paper_weights():
    """L = sum_k lambda_k D^(k) with the paper's five-prefix weightings (Sec. 5, App. G.2)."""
    layer, W_bits, H = _case(192, 512, 5, "f16", seed=21)
    lin, W, Hd = _device(layer, W_bits, H)
    for name, lam in oracle_pins._paper_loss_weights().items():
        d = lin.wmse(W, Hd, lam).cpu().numpy()
        ref = _check(layer, W_bits, H, d[:5], name)
        want = oracle.dbyd_loss(d[:5], lam)
        assert abs(d[5] - want) <= 1e-15 * abs(want), (name, d[5], want)
        assert abs(d[5] - oracle.dbyd_loss(ref, lam)) <= BOUND_REL * oracle.dbyd_loss(ref, lam)


def test_repeatable_and_empty():
    layer, W_bits, H = _case(128, 256, 2, "bf16", seed=5)
    lin, W, Hd = _device(layer, W_bits, H)
    a, b = lin.wmse(W, Hd), lin.wmse(W, Hd)
    assert torch.equal(a, b)                                # fixed summation order
    # a layer without rows: every D (and L) is zero, nothing else is read
    z = torch.full((3,), 7.0, dtype=torch.float64, device="cuda")
    aq.aq_wmse(aq.Layout.make(0, 256, 2), None, None, None, None, None, aq.AQ_F32, [0.5, 0.5],
               z, None, 0)
    assert torch.equal(z.cpu(), torch.zeros(3, dtype=torch.float64))


def test_full_size_attn_4096():
    """The 4096 x 4096 layer of the benchmark, four prefixes, against the fp64 oracle."""
    layer, W_bits, H = _case(4096, 4096, 4, "f16", seed=41)
    lin, W, Hd = _device(layer, W_bits, H)
    _check(layer, W_bits, H, lin.wmse(W, Hd).cpu().numpy(), "4096")


def test_wmse_argument_errors():
    layer, W_bits, H = _case(64, 256, 2, "f16", seed=6)
    lin, W, Hd = _device(layer, W_bits, H)
    lib = aq.lib()
    d = torch.empty(3, dtype=torch.float64, device="cuda")
    nbytes = aq.wmse_workspace_bytes(lin.layout)
    ws = aq.workspace(nbytes)
    call = lambda L, hdt=aq.AQ_F32, d_ptr=d.data_ptr(), wsb=nbytes: lib.aq_wmse(
        ctypes.byref(L), W.data_ptr(), lin.planes.data_ptr(), lin.books.data_ptr(),
        lin.scales.data_ptr(), Hd.data_ptr(), hdt, None, d_ptr, ws.data_ptr(), wsb, None)
    assert call(lin.layout, hdt=aq.AQ_F16) == aq.AQ_ERR_INVALID_ARG
    assert call(lin.layout, d_ptr=None) == aq.AQ_ERR_INVALID_ARG
    assert call(lin.layout, d_ptr=d.data_ptr() + 4) == aq.AQ_ERR_ALIGNMENT
    assert call(lin.layout, wsb=nbytes - 16) == aq.AQ_ERR_WORKSPACE
    assert call(lin.layout) == aq.AQ_OK
    assert aq.aq_workspace_status(ws) == aq.AQ_OK
