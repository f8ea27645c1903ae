"""Python binding of libaq, the GB300 multi-bitwidth additive-codebook library (include/aq.h).

Argument marshalling only: every function forwards to the C entry point of the same name in
libaq.so, passing device pointers of torch tensors and the current CUDA stream. All the
arithmetic runs in the library's CUDA kernels; there is no Python or CPU fallback, and the
functions raise if the library is missing.
"""
import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libaq.so")

AQ_OK, AQ_ERR_INVALID_ARG, AQ_ERR_UNSUPPORTED, AQ_ERR_ALIGNMENT = 0, 1, 2, 3
AQ_ERR_CUDA, AQ_ERR_TIMEOUT, AQ_ERR_WORKSPACE = 4, 5, 6
AQ_F16, AQ_BF16, AQ_F32 = 0, 1, 2
AQ_LAYOUT_STATIC_WEIGHTS = 1
DTYPES = {"f16": AQ_F16, "bf16": AQ_BF16, "f32": AQ_F32}
TORCH_DTYPES = {AQ_F16: torch.float16, AQ_BF16: torch.bfloat16, AQ_F32: torch.float32}

# Every entry point that include/aq.h declares.
EXPORTS = ["aq_abi_version", "aq_status_string", "aq_last_error", "aq_plane_bytes", "aq_packed_bytes", "aq_pack",
           "aq_decode", "aq_gemv_workspace_bytes", "aq_gemv", "aq_gemm_workspace_bytes",
           "aq_gemm", "aq_workspace_init", "aq_workspace_status", "aq_gemv_static_scratch",
           "aq_gemv_static_scratch_status",
           "aq_gemv_refine", "aq_store_create", "aq_store_set_prefix", "aq_store_prefix",
           "aq_store_planes", "aq_store_books", "aq_store_scales", "aq_store_device_bytes",
           "aq_store_destroy", "aq_wmse_workspace_bytes", "aq_wmse", "aq_beam_workspace_bytes",
           "aq_beam_search", "aq_selftest_wait", "aq_selftest_read", "aq_gemv_group_workspace_bytes",
           "aq_gemv_group"]


class AQError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        msg = "%s failed: %s (status %d)" % (where, status_string(status), status)
        if status == AQ_ERR_CUDA:
            msg += ": " + lib().aq_last_error().decode()
        super().__init__(msg)


class Layout(ctypes.Structure):
    """struct aq_layout."""
    _fields_ = [("out_features", ctypes.c_int32), ("in_features", ctypes.c_int32),
                ("group_size", ctypes.c_int32), ("num_books", ctypes.c_int32),
                ("code_bits", ctypes.c_int32), ("book_dtype", ctypes.c_int32),
                ("scale_dtype", ctypes.c_int32), ("flags", ctypes.c_int32)]

    @classmethod
    def make(cls, out, inp, M, B=8, G=8, book_dtype="f16", scale_dtype="f16", flags=0):
        return cls(out, inp, G, M, B, DTYPES[book_dtype], DTYPES[scale_dtype], flags)


_lib = None


def lib():
    """Load libaq.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libaq.so is not built; run __graft_entry__.build() or "
                               "python paper_2606_12876_gb300/build.py")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        lp = ctypes.POINTER(Layout)
        sig = {
            "aq_abi_version": (i32, []),
            "aq_status_string": (ctypes.c_char_p, [i32]),
            "aq_last_error": (ctypes.c_char_p, []),
            "aq_plane_bytes": (sz, [lp]),
            "aq_packed_bytes": (sz, [lp, i32]),
            "aq_pack": (i32, [lp, vp, vp, vp]),
            "aq_decode": (i32, [lp, i32, vp, vp, vp, vp, vp]),
            "aq_gemv_workspace_bytes": (sz, [lp, i32]),
            "aq_gemv": (i32, [lp, i32, vp, vp, vp, vp, i32, i32, vp, i32, vp, sz, vp]),
            "aq_gemm_workspace_bytes": (sz, [lp, i32]),
            "aq_gemm": (i32, [lp, i32, vp, vp, vp, vp, i32, i32, vp, i32, vp, sz, vp]),
            "aq_workspace_init": (i32, [vp, sz, vp]),
            "aq_workspace_status": (i32, [vp, vp]),
            "aq_gemv_static_scratch": (i32, [lp, i32, vp, vp, vp, vp, i32, i32, vp, i32, vp]),
            "aq_gemv_static_scratch_status": (i32, [vp]),
            "aq_gemv_refine": (i32, [lp, i32, vp, vp, vp, vp, i32, i32, vp, vp, i32, vp, sz, vp]),
            "aq_store_create": (i32, [lp, ctypes.POINTER(vp)]),
            "aq_store_set_prefix": (i32, [vp, i32, vp, vp, vp, vp]),
            "aq_store_prefix": (i32, [vp]),
            "aq_store_planes": (vp, [vp]),
            "aq_store_books": (vp, [vp]),
            "aq_store_scales": (vp, [vp]),
            "aq_store_device_bytes": (sz, [vp]),
            "aq_store_destroy": (i32, [vp]),
            "aq_wmse_workspace_bytes": (sz, [lp]),
            "aq_beam_workspace_bytes": (sz, [lp]),
            "aq_beam_search": (i32, [lp, vp, vp, vp, vp, vp, i32, ctypes.POINTER(ctypes.c_double),
                                     i32, vp, vp, sz, vp]),
            "aq_selftest_wait": (i32, [vp, sz, vp]),
            "aq_selftest_read": (i32, [vp, sz, vp, vp]),
            "aq_gemv_group_workspace_bytes": (sz, [i32, lp, i32]),
            "aq_gemv_group": (i32, [i32, lp, i32, ctypes.POINTER(vp), ctypes.POINTER(vp),
                                    ctypes.POINTER(vp), vp, i32, i32, ctypes.POINTER(vp), i32,
                                    vp, sz, vp]),
            "aq_wmse": (i32, [lp, vp, vp, vp, vp, vp, i32, ctypes.POINTER(ctypes.c_double), vp,
                              vp, sz, vp]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype, fn.argtypes = res, args
        _lib = L
    return _lib


def status_string(status):
    return lib().aq_status_string(int(status)).decode()


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


# The current stream as a raw handle, without building a Stream object per call (torch's
# accessor when present).
_raw_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream(stream):
    if stream is None:
        if _raw_stream is not None:
            return _raw_stream(torch.cuda.current_device())
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status, where):
    if status != AQ_OK:
        raise AQError(status, where)


def abi_version():
    return lib().aq_abi_version()


def plane_bytes(layout):
    return lib().aq_plane_bytes(ctypes.byref(layout))


def packed_bytes(layout, m):
    return lib().aq_packed_bytes(ctypes.byref(layout), m)


def gemv_workspace_bytes(layout, batch):
    return lib().aq_gemv_workspace_bytes(ctypes.byref(layout), batch)


def gemm_workspace_bytes(layout, tokens):
    return lib().aq_gemm_workspace_bytes(ctypes.byref(layout), tokens)


def aq_pack(layout, codes, planes, stream=None):
    _check(lib().aq_pack(ctypes.byref(layout), _ptr(codes), _ptr(planes), _stream(stream)),
           "aq_pack")


def aq_decode(layout, m, planes, books, scales, w, stream=None):
    _check(lib().aq_decode(ctypes.byref(layout), m, _ptr(planes), _ptr(books), _ptr(scales),
                           _ptr(w), _stream(stream)), "aq_decode")


def aq_gemv(layout, m, planes, books, scales, x, x_dtype, batch, y, y_dtype, workspace,
            workspace_bytes=None, stream=None):
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(lib().aq_gemv(ctypes.byref(layout), m, _ptr(planes), _ptr(books), _ptr(scales),
                         _ptr(x), x_dtype, batch, _ptr(y), y_dtype, _ptr(workspace),
                         workspace_bytes, _stream(stream)), "aq_gemv")


def aq_gemv_refine(layout, m, planes, books, scales, x, x_dtype, batch, y_prev, y, y_dtype,
                   workspace, workspace_bytes=None, stream=None):
    """y = y_prev + x (s o C_{m-1}[b_{m-1}])^T (y_prev None: zero); reads plane m-1 only."""
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(lib().aq_gemv_refine(ctypes.byref(layout), m, _ptr(planes), _ptr(books), _ptr(scales),
                                _ptr(x), x_dtype, batch, _ptr(y_prev), _ptr(y), y_dtype,
                                _ptr(workspace), workspace_bytes, _stream(stream)),
           "aq_gemv_refine")


def aq_gemm(layout, m, planes, books, scales, x, x_dtype, tokens, y, y_dtype, workspace,
            workspace_bytes=None, stream=None):
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    _check(lib().aq_gemm(ctypes.byref(layout), m, _ptr(planes), _ptr(books), _ptr(scales),
                         _ptr(x), x_dtype, tokens, _ptr(y), y_dtype, _ptr(workspace),
                         workspace_bytes, _stream(stream)), "aq_gemm")


def aq_gemv_static_scratch(layout, m, planes, books, scales, x, x_dtype, batch, y, y_dtype,
                           stream=None):
    """aq_gemv without a workspace: scratch comes from the library's fixed device buffer."""
    _check(lib().aq_gemv_static_scratch(ctypes.byref(layout), m, _ptr(planes), _ptr(books),
                                        _ptr(scales), _ptr(x), x_dtype, batch, _ptr(y), y_dtype,
                                        _stream(stream)), "aq_gemv_static_scratch")


def aq_gemv_static_scratch_status(stream=None):
    """The device-side status of the aq_gemv_static_scratch calls on the current device
    (synchronises the stream; clears the status)."""
    return lib().aq_gemv_static_scratch_status(_stream(stream))


def aq_store_create(layout):
    """An empty prefix store for layout on the current device (an opaque handle, an int)."""
    h = ctypes.c_void_p()
    _check(lib().aq_store_create(ctypes.byref(layout), ctypes.byref(h)), "aq_store_create")
    return h.value


def aq_store_set_prefix(store, m, src_planes, src_books, src_scales, stream=None):
    """Make planes/codebooks 0..m-1 resident (copies enqueued on the stream when raising; the
    device is synchronised when lowering). Sources: tensors or addresses, host or device."""
    _check(lib().aq_store_set_prefix(store, m, _ptr(src_planes), _ptr(src_books),
                                     _ptr(src_scales), _stream(stream)), "aq_store_set_prefix")


def aq_store_prefix(store):
    return lib().aq_store_prefix(store)


def aq_store_planes(store):
    return lib().aq_store_planes(store)


def aq_store_books(store):
    return lib().aq_store_books(store)


def aq_store_scales(store):
    return lib().aq_store_scales(store)


def aq_store_device_bytes(store):
    return lib().aq_store_device_bytes(store)


def aq_store_destroy(store):
    _check(lib().aq_store_destroy(store), "aq_store_destroy")


def wmse_workspace_bytes(layout):
    return lib().aq_wmse_workspace_bytes(ctypes.byref(layout))


def aq_wmse(layout, w, planes, books, scales, h, h_dtype, lam, d, workspace,
            workspace_bytes=None, stream=None):
    """d[k-1] = tr[(W - W^(k)) H (W - W^(k))^T] / d_out for k = 1..M; with lam (M host
    floats) also d[M] = sum_k lam[k-1] d[k-1]."""
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    lam_arr = None
    if lam is not None:
        lam_arr = (ctypes.c_double * len(lam))(*[float(v) for v in lam])
    _check(lib().aq_wmse(ctypes.byref(layout), _ptr(w), _ptr(planes), _ptr(books), _ptr(scales),
                         _ptr(h), h_dtype, lam_arr, _ptr(d), _ptr(workspace), workspace_bytes,
                         _stream(stream)), "aq_wmse")


def beam_workspace_bytes(layout):
    return lib().aq_beam_workspace_bytes(ctypes.byref(layout))


def aq_beam_search(layout, w, codes, books, scales, h, h_dtype, lam, beam, codes_out, workspace,
                   workspace_bytes=None, stream=None):
    """New codes [d_out][d_in/8][M] (into codes_out) from a beam search of width `beam` per
    group over the books, minimising sum_k lam[k-1] e^(k) S e^(k)^T of the group's row with the
    other groups at their current codes (lam: M host floats, or None for all ones)."""
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    lam_arr = None
    if lam is not None:
        lam_arr = (ctypes.c_double * len(lam))(*[float(v) for v in lam])
    _check(lib().aq_beam_search(ctypes.byref(layout), _ptr(w), _ptr(codes), _ptr(books),
                                _ptr(scales), _ptr(h), h_dtype, lam_arr, int(beam),
                                _ptr(codes_out), _ptr(workspace), workspace_bytes,
                                _stream(stream)), "aq_beam_search")


def aq_workspace_init(workspace, nbytes=None, stream=None):
    if nbytes is None:
        nbytes = workspace.numel() * workspace.element_size()
    _check(lib().aq_workspace_init(_ptr(workspace), nbytes, _stream(stream)), "aq_workspace_init")


def gemv_group_workspace_bytes(layouts, batch):
    arr = (Layout * len(layouts))(*layouts)
    return lib().aq_gemv_group_workspace_bytes(len(layouts), arr, batch)


def aq_gemv_group(layouts, m, planes, books, scales, x, x_dtype, batch, ys, y_dtype, workspace,
                  workspace_bytes=None, stream=None):
    """The GEMVs of several layers that share the activations x (one call of aq_gemv_group)."""
    n = len(layouts)
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    vp = ctypes.c_void_p
    arr = (Layout * n)(*layouts)
    _check(lib().aq_gemv_group(n, arr, m, (vp * n)(*[_ptr(p) for p in planes]),
                               (vp * n)(*[_ptr(b) for b in books]),
                               (vp * n)(*[_ptr(s) for s in scales]), _ptr(x), x_dtype, batch,
                               (vp * n)(*[_ptr(y) for y in ys]), y_dtype, _ptr(workspace),
                               workspace_bytes, _stream(stream)), "aq_gemv_group")


def aq_selftest_read(src, nbytes, sink, stream=None):
    """Read probe: XOR of the 32-bit words of the first nbytes of src folded into sink[0]."""
    _check(lib().aq_selftest_read(_ptr(src), nbytes, _ptr(sink), _stream(stream)),
           "aq_selftest_read")


def aq_workspace_status(workspace, stream=None):
    """Synchronises the stream; returns the device-side status recorded in the workspace."""
    return lib().aq_workspace_status(_ptr(workspace), _stream(stream))


def workspace(nbytes, device="cuda"):
    """A zero-filled workspace tensor of at least nbytes (16-byte aligned by the allocator)."""
    return torch.zeros(max(16, (nbytes + 15) // 16 * 16), dtype=torch.uint8, device=device)
