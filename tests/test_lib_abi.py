"""The C-ABI library without a GPU: it loads, exports what include/aq.h declares, answers size
queries that agree with the oracle's packed layout, and rejects bad arguments on the host
(no compute call is made here)."""
import ctypes
import os
import re

import numpy as np
import pytest

import aq_testutil
import oracle
import paper_2606_12876_gb300 as aq
import workloads

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "aq.h")
FAKE = 1 << 20          # an aligned non-null address; never dereferenced by these tests


@pytest.fixture(scope="module", autouse=True)
def built():
    aq_testutil.ensure_built()


def header_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:aq_status|size_t|int|const char\*|void\*)\s+(aq_\w+)\s*\(",
                                 text, flags=re.M)))


def test_every_declared_symbol_is_exported():
    names = header_functions()
    assert len(names) >= 12
    L = ctypes.CDLL(aq.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert sorted(aq.EXPORTS) == names


def test_version_and_status_strings():
    assert aq.abi_version() == 1
    for s in range(7):
        assert aq.status_string(s) and aq.status_string(s) != "unknown status"
    assert aq.status_string(99) == "unknown status"


@pytest.mark.parametrize("out,inp,M,B", [(1, 8, 1, 8), (37, 560, 3, 8), (64, 256, 4, 8),
                                          (50, 136, 2, 16), (4096, 4096, 4, 8), (37, 560, 3, 4)])
def test_packed_sizes_match_oracle_layout(out, inp, M, B):
    L = aq.Layout.make(out, inp, M, B=B)
    layer = dict(out=out, **{"in": inp}, G=8, M=M, B=B,
                 codes=np.zeros((out, inp // 8, M), np.uint8 if B <= 8 else np.uint16))
    total = oracle.pack(layer).size
    assert aq.plane_bytes(L) * M == total
    for m in range(1, M + 1):
        assert aq.packed_bytes(L, m) == m * aq.plane_bytes(L)
    assert aq.packed_bytes(L, 0) == 0 and aq.packed_bytes(L, M + 1) == 0


def test_gemv_workspace_covers_partials():
    L = aq.Layout.make(4096, 4096, 4)
    # 16 slices x batch x 4096 rows of fp32 partials, plus status and counters
    assert aq.gemv_workspace_bytes(L, 1) >= 16 * 4096 * 4
    assert aq.gemv_workspace_bytes(L, 16) >= 16 * 16 * 4096 * 4
    assert aq.gemv_workspace_bytes(L, 17) == 0


def _lay(**kw):
    base = dict(out=64, inp=256, M=4, B=8, G=8, book_dtype="f16", scale_dtype="f16")
    base.update(kw)
    return aq.Layout.make(**base)


@pytest.mark.parametrize("kw,status", [
    (dict(G=4), aq.AQ_ERR_UNSUPPORTED), (dict(B=5), aq.AQ_ERR_UNSUPPORTED),
    (dict(B=12), aq.AQ_ERR_UNSUPPORTED),
    (dict(B=17), aq.AQ_ERR_INVALID_ARG), (dict(M=9), aq.AQ_ERR_UNSUPPORTED),
    (dict(M=0), aq.AQ_ERR_INVALID_ARG), (dict(inp=260), aq.AQ_ERR_INVALID_ARG),
    (dict(inp=0), aq.AQ_ERR_INVALID_ARG), (dict(out=-1), aq.AQ_ERR_INVALID_ARG),
])
def test_layout_rejected(kw, status):
    L = _lay(**kw)
    assert aq.plane_bytes(L) == 0
    rc = aq.lib().aq_decode(ctypes.byref(L), 1, FAKE, FAKE, FAKE, FAKE, None)
    assert rc == status


def test_bad_dtype_rejected():
    L = _lay()
    L.book_dtype = 7
    assert aq.lib().aq_decode(ctypes.byref(L), 1, FAKE, FAKE, FAKE, FAKE, None) == aq.AQ_ERR_INVALID_ARG


def _gemv(L, m=1, planes=FAKE, x=FAKE, x_dt=aq.AQ_F16, batch=1, y=FAKE, y_dt=aq.AQ_F16,
          ws=FAKE, ws_bytes=None):
    if ws_bytes is None:
        ws_bytes = aq.gemv_workspace_bytes(L, max(1, min(batch, 16)))
    return aq.lib().aq_gemv(ctypes.byref(L), m, planes, FAKE, FAKE, x, x_dt, batch, y, y_dt, ws,
                            ws_bytes, None)


def test_gemv_argument_errors():
    L = _lay()
    assert _gemv(L, m=0) == aq.AQ_ERR_INVALID_ARG
    assert _gemv(L, m=5) == aq.AQ_ERR_INVALID_ARG
    assert _gemv(L, batch=17) == aq.AQ_ERR_INVALID_ARG
    assert _gemv(L, batch=-1) == aq.AQ_ERR_INVALID_ARG
    assert _gemv(L, x_dt=aq.AQ_F32) == aq.AQ_ERR_INVALID_ARG
    assert _gemv(L, y_dt=9) == aq.AQ_ERR_INVALID_ARG
    assert _gemv(L, planes=None) == aq.AQ_ERR_INVALID_ARG
    assert _gemv(L, x=FAKE + 2) == aq.AQ_ERR_ALIGNMENT
    assert _gemv(L, ws=None) == aq.AQ_ERR_WORKSPACE
    assert _gemv(L, ws_bytes=aq.gemv_workspace_bytes(L, 1) - 4) == aq.AQ_ERR_WORKSPACE
    # empty work is a successful no-op that touches nothing
    assert _gemv(L, batch=0, planes=None, x=None, y=None, ws=None) == aq.AQ_OK
    assert _gemv(_lay(out=0), planes=None, x=None, y=None, ws=None) == aq.AQ_OK


def test_decode_and_pack_argument_errors():
    L = _lay()
    lib = aq.lib()
    assert lib.aq_decode(ctypes.byref(L), 0, FAKE, FAKE, FAKE, FAKE, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_decode(ctypes.byref(L), 1, FAKE, None, FAKE, FAKE, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_decode(ctypes.byref(L), 1, FAKE, FAKE, FAKE + 8, FAKE, None) == aq.AQ_ERR_ALIGNMENT
    assert lib.aq_pack(ctypes.byref(L), None, FAKE, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_pack(None, FAKE, FAKE, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_workspace_init(None, 16, None) == aq.AQ_ERR_INVALID_ARG


def test_store_argument_errors_on_the_host():
    """Checks a prefix store makes before any CUDA call (no device needed)."""
    lib = aq.lib()
    h = ctypes.c_void_p()
    assert lib.aq_store_create(None, ctypes.byref(h)) == aq.AQ_ERR_INVALID_ARG
    assert h.value is None
    assert lib.aq_store_create(ctypes.byref(_lay()), None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_store_create(ctypes.byref(_lay(G=4)), ctypes.byref(h)) == aq.AQ_ERR_UNSUPPORTED
    assert lib.aq_store_create(ctypes.byref(_lay(M=0)), ctypes.byref(h)) == aq.AQ_ERR_INVALID_ARG
    assert h.value is None
    assert lib.aq_store_set_prefix(None, 1, FAKE, FAKE, FAKE, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_store_prefix(None) == 0 and lib.aq_store_device_bytes(None) == 0
    assert lib.aq_store_planes(None) is None and lib.aq_store_books(None) is None
    assert lib.aq_store_scales(None) is None
    assert lib.aq_store_destroy(None) == aq.AQ_OK


def test_wmse_sizes_and_argument_errors_on_the_host():
    L = aq.Layout.make(4096, 4096, 4)
    # status block, the folded H in bf16, E_k of the four prefixes in bf16, one fp32 partial
    # per CTA of a pass and prefix (2 CTAs per 256 x 256 tile: 16 x 16 tiles)
    assert aq.wmse_workspace_bytes(L) == (1024 + 4096 * 4096 * 2 + 4 * 4096 * 4096 * 2
                                          + 2 * 16 * 16 * 4 * 4)
    lib = aq.lib()
    d8 = FAKE
    call = lambda L, hdt=aq.AQ_F32, d=d8, ws=FAKE, wsb=None: lib.aq_wmse(
        ctypes.byref(L) if L is not None else None, FAKE, FAKE, FAKE, FAKE, FAKE, hdt, None, d,
        ws, aq.wmse_workspace_bytes(L) if wsb is None and L is not None else (wsb or 0), None)
    assert call(None, wsb=0) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), hdt=aq.AQ_F16) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), d=None) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), d=FAKE + 4) == aq.AQ_ERR_ALIGNMENT
    assert call(_lay(), ws=None) == aq.AQ_ERR_WORKSPACE
    assert call(_lay(), wsb=aq.wmse_workspace_bytes(_lay()) - 16) == aq.AQ_ERR_WORKSPACE
    assert call(_lay(), ws=FAKE + 8) == aq.AQ_ERR_ALIGNMENT


def test_beam_sizes_and_argument_errors_on_the_host():
    L = aq.Layout.make(4096, 4096, 4)
    # status block, S in fp32, then E_k and E_k S of the four prefixes in fp32
    assert aq.beam_workspace_bytes(L) == 256 + 4096 * 4096 * 4 + 2 * 4 * 4096 * 4096 * 4
    lib = aq.lib()

    def call(L, hdt=aq.AQ_F32, lam=None, K=4, out=FAKE, ws=FAKE, wsb=None):
        lam_arr = None if lam is None else (ctypes.c_double * len(lam))(*lam)
        return lib.aq_beam_search(
            ctypes.byref(L) if L is not None else None, FAKE, FAKE, FAKE, FAKE, FAKE, hdt,
            lam_arr, K, out, ws,
            aq.beam_workspace_bytes(L) if wsb is None and L is not None else (wsb or 0), None)
    assert call(None, wsb=0) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), hdt=aq.AQ_F16) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), K=0) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), K=17) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), lam=[1.0, -0.5, 1.0, 1.0]) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), lam=[1.0, float("nan"), 1.0, 1.0]) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(B=16)) == aq.AQ_ERR_UNSUPPORTED
    assert call(_lay(), out=None) == aq.AQ_ERR_INVALID_ARG
    assert call(_lay(), out=FAKE + 1) == aq.AQ_ERR_ALIGNMENT
    assert call(_lay(), ws=None) == aq.AQ_ERR_WORKSPACE
    assert call(_lay(), wsb=aq.beam_workspace_bytes(_lay()) - 4) == aq.AQ_ERR_WORKSPACE
    assert call(_lay(), ws=FAKE + 8) == aq.AQ_ERR_ALIGNMENT
    assert call(_lay(out=0), ws=None) == aq.AQ_OK      # nothing to update


def _x16(tokens):
    """Offset of the fp16 activation copy: status block, then one float per token."""
    return 256 + (tokens * 4 + 255) // 256 * 256


def test_gemm_workspace_sizes():
    """Status block + per-token activation factors + fp16 activation copy; from 2048 tokens
    (two or more books) also room for W_m decoded once in fp16."""
    L = aq.Layout.make(300, 520, 4)
    assert aq.gemm_workspace_bytes(L, 2047) == _x16(2047) + 2047 * 520 * 2
    off = (_x16(2048) + 2048 * 520 * 2 + 1023) // 1024 * 1024
    assert aq.gemm_workspace_bytes(L, 2048) == off + 300 * 520 * 2
    L1 = aq.Layout.make(300, 520, 1)
    assert aq.gemm_workspace_bytes(L1, 4096) == _x16(4096) + 4096 * 520 * 2


def test_gemm_workspace_for_4bit_codes():
    """4-bit layouts always decode W_m into the workspace first."""
    L = aq.Layout.make(300, 520, 4, B=4)
    off = (_x16(40) + 40 * 520 * 2 + 1023) // 1024 * 1024
    assert aq.gemm_workspace_bytes(L, 40) == off + 300 * 520 * 2
    assert aq.plane_bytes(L) == 320 * 96 // 2


def test_selftest_wait_argument_errors_on_the_host():
    lib = aq.lib()
    assert lib.aq_selftest_wait(None, 256, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_selftest_wait(FAKE, 16, None) == aq.AQ_ERR_WORKSPACE
    assert lib.aq_selftest_wait(FAKE + 8, 256, None) == aq.AQ_ERR_ALIGNMENT


def test_selftest_read_argument_errors_on_the_host():
    lib = aq.lib()
    assert lib.aq_selftest_read(FAKE, 1024, None, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_selftest_read(None, 1024, FAKE, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_selftest_read(FAKE + 8, 1024, FAKE, None) == aq.AQ_ERR_ALIGNMENT
    assert lib.aq_selftest_read(FAKE, 1000, FAKE, None) == aq.AQ_ERR_ALIGNMENT
    assert lib.aq_selftest_read(FAKE, 1024, FAKE + 2, None) == aq.AQ_ERR_ALIGNMENT


def test_gemv_workspace_follows_the_kernel_choice():
    """Batch 5..8: one partial plane per (slice, book, token) when the eight-token table kernel
    serves the layer (at least 4560 (slice, book, row block) items at the largest prefix it
    takes, six books), else one per (slice, token)."""
    big = aq.Layout.make(1000, 8200, 6)            # 33 slices x 6 books x 32 row blocks
    assert aq.gemv_workspace_bytes(big, 8) == 256 + 33 * 8 * 6 * 1024 * 4
    small = aq.Layout.make(300, 1032, 4)           # 5 slices x 4 books x 10 row blocks
    assert aq.gemv_workspace_bytes(small, 8) == 256 + 5 * 8 * 320 * 4
    assert aq.gemv_workspace_bytes(big, 16) == 256 + 33 * 16 * 1024 * 4


def test_gemv_group_workspace_and_argument_errors_on_the_host():
    """aq_gemv_group: the workspace is the layers' aq_gemv workspaces one after the other, each
    rounded up to 256 bytes; host-side argument errors launch nothing."""
    Ls = [aq.Layout.make(4096, 4096, 4), aq.Layout.make(1024, 4096, 4), aq.Layout.make(1000, 4096, 2)]
    want = sum((aq.gemv_workspace_bytes(L, 1) + 255) // 256 * 256 for L in Ls)
    assert aq.gemv_group_workspace_bytes(Ls, 1) == want
    lib = aq.lib()
    vp = ctypes.c_void_p
    arr3 = (aq.Layout * 3)(*Ls)
    ptrs = (vp * 3)(FAKE, FAKE, FAKE)
    args = lambda n, layouts, m=1: (n, layouts, m, ptrs, ptrs, ptrs, FAKE, aq.AQ_F16, 1, ptrs,
                                    aq.AQ_F16, FAKE, 1 << 30, None)
    assert lib.aq_gemv_group(*args(0, arr3)) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_gemv_group(*args(5, (aq.Layout * 5)(*(Ls + Ls[:2])))) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_gemv_group(*args(3, arr3, m=3)) == aq.AQ_ERR_INVALID_ARG      # m > M of layer 2
    other = (aq.Layout * 2)(Ls[0], aq.Layout.make(1024, 2048, 4))               # in differs
    assert lib.aq_gemv_group(*args(2, other)) == aq.AQ_ERR_INVALID_ARG
    bf = (aq.Layout * 2)(Ls[0], aq.Layout.make(1024, 4096, 4, book_dtype="bf16"))
    assert lib.aq_gemv_group(*args(2, bf)) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_gemv_group(3, arr3, 1, None, ptrs, ptrs, FAKE, aq.AQ_F16, 1, ptrs, aq.AQ_F16,
                             FAKE, 1 << 30, None) == aq.AQ_ERR_INVALID_ARG
    assert lib.aq_gemv_group(*(args(3, arr3)[:11] + (FAKE, 16, None))) == aq.AQ_ERR_WORKSPACE
