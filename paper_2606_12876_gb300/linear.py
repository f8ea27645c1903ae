"""AQLinear: one additive-codebook linear layer resident on the GPU, served at any prefix m.

The layer is stored once (AQLMFormat(C, b, s) of Alg. 1: M codebooks, codes, per-row scales)
and evaluated with the first m codebooks chosen per call (Sec. 5). A layer either holds all M
codebooks in torch device memory, or (from_host) holds only a resident prefix in a libaq store
that loads further codebooks from host memory at run time. All work is done by libaq through
the binding in this package.
"""
import weakref

import numpy as np
import torch

from . import (AQ_BF16, AQ_F16, AQ_F32, AQ_LAYOUT_STATIC_WEIGHTS, DTYPES, TORCH_DTYPES, Layout,
               aq_decode, aq_gemm, aq_gemv_group, gemv_group_workspace_bytes,
               aq_gemv, aq_gemv_refine, aq_pack, aq_store_books, aq_store_create, aq_wmse,
               wmse_workspace_bytes, aq_workspace_init,
               aq_store_device_bytes, aq_store_planes, aq_store_scales, aq_store_set_prefix,
               gemm_workspace_bytes, gemv_workspace_bytes, lib, packed_bytes,
               workspace, _stream)


def _destroy_store(store):
    lib().aq_store_destroy(store)


def _u16_to_device(a, device):
    a = np.ascontiguousarray(a, dtype=np.uint16)
    return torch.from_numpy(a.view(np.int16)).to(device)


class AQLinear:
    """Packed planes, codebooks and scales of one layer on `device`.

    books: [M][2^B][8] fp16/bf16 bit patterns (uint16), B = 4, 8 or 16; codes: (out, in/8, M)
    uint8 (B <= 8) or uint16;
    scales: [out] bit patterns. The natural codes are packed on the GPU by aq_pack. After
    packing the stream is synchronised and the layout is marked AQ_LAYOUT_STATIC_WEIGHTS: the
    layer's weights are read-only from then on, so calls may prefetch them early.
    """

    def __init__(self, books, codes, scales, book_dtype="f16", scale_dtype="f16",
                 device="cuda", keep_codes=False):
        out, ng, M = codes.shape
        B = int(np.asarray(books).shape[1]).bit_length() - 1     # books: [M][2^B][8]
        self.layout = Layout.make(out, ng * 8, M, B=B, book_dtype=book_dtype,
                                  scale_dtype=scale_dtype)
        self.out, self.inp, self.M, self.B = out, ng * 8, M, B
        self.device = torch.device(device)
        self.book_dtype, self.scale_dtype = book_dtype, scale_dtype
        self.books = _u16_to_device(books, self.device)
        self.scales = _u16_to_device(scales, self.device)
        codes_t = torch.from_numpy(np.ascontiguousarray(codes).view(
            np.int8 if B <= 8 else np.int16)).to(self.device)
        self.planes = torch.empty(packed_bytes(self.layout, M), dtype=torch.uint8,
                                  device=self.device)
        aq_pack(self.layout, codes_t, self.planes)
        torch.cuda.current_stream(self.device).synchronize()
        self.layout.flags = AQ_LAYOUT_STATIC_WEIGHTS
        self.codes = codes_t if keep_codes else None
        self._ws = {}
        self.store, self.resident = None, M

    @classmethod
    def from_layer(cls, layer, device="cuda", keep_codes=False):
        """From a workloads.make_layer() dict."""
        return cls(layer["books"], layer["codes"], layer["scales"], layer["book_dtype"],
                   layer["scale_dtype"], device, keep_codes)

    def to_host(self, pin=True):
        """The packed layer in host memory, the form a deployment keeps outside the GPU: a dict
        of the layout, the planes of all M codebooks (uint8), the codebooks and the scales
        (int16 bit patterns), and the dtype names; page-locked when pin is true, so that
        loading from it runs as asynchronous copies."""
        if self.store is not None:
            raise TypeError("to_host needs a layer that holds all its codebooks")
        t = lambda a: a.cpu().pin_memory() if pin else a.cpu()
        layout = Layout(*[getattr(self.layout, f) for f, _ in Layout._fields_])
        return dict(layout=layout, planes=t(self.planes), books=t(self.books),
                    scales=t(self.scales), book_dtype=self.book_dtype,
                    scale_dtype=self.scale_dtype)

    @classmethod
    def from_host(cls, host, m, device="cuda"):
        """A layer whose device memory holds only the first m codebooks (a libaq store); more
        are loaded from `host` (a to_host() dict, kept referenced) by set_prefix. Calls accept
        prefixes up to the resident one."""
        self = cls.__new__(cls)
        L = host["layout"]
        self.layout = Layout(*[getattr(L, f) for f, _ in Layout._fields_])
        self.layout.flags = AQ_LAYOUT_STATIC_WEIGHTS
        self.out, self.inp, self.M, self.B = (L.out_features, L.in_features, L.num_books,
                                              L.code_bits)
        self.device = torch.device(device)
        self.book_dtype, self.scale_dtype = host["book_dtype"], host["scale_dtype"]
        with torch.cuda.device(self.device):
            self.store = aq_store_create(self.layout)
        self._finalizer = weakref.finalize(self, _destroy_store, self.store)
        self._host = host
        self.planes = aq_store_planes(self.store)
        self.books = aq_store_books(self.store)
        self.scales = aq_store_scales(self.store)
        self.codes, self._ws, self.resident = None, {}, 0
        self.set_prefix(m)
        return self

    def set_prefix(self, m):
        """Raise or lower the resident prefix of a from_host layer to m (0..M). Raising copies
        planes and codebooks on the current stream, so later work on that stream sees them;
        lowering releases the dropped planes' memory once the work enqueued on the current
        stream so far has finished (nothing waits for it; work reading the dropped planes must
        have been enqueued on this stream)."""
        if self.store is None:
            raise TypeError("set_prefix needs a layer made by from_host")
        h = self._host
        with torch.cuda.device(self.device):
            aq_store_set_prefix(self.store, m, h["planes"], h["books"], h["scales"])
        self.resident = m

    def device_bytes(self):
        """Device memory held for the layer's weights (scales, codebooks, resident planes, and
        for a from_host layer dropped planes whose release still waits for their stream)."""
        if self.store is not None:
            return aq_store_device_bytes(self.store)
        return sum(t.numel() * t.element_size() for t in (self.planes, self.books, self.scales))

    def close(self):
        """Release a from_host layer's device memory now (synchronises the device)."""
        if self.store is not None:
            self._finalizer()
            self.store, self.planes, self.books, self.scales, self.resident = None, None, None, None, 0

    def _check_m(self, m):
        # A prefix beyond the resident one would read device memory that is not mapped.
        if not 1 <= m <= self.resident:
            raise ValueError("prefix m=%d outside 1..%d (resident codebooks)" % (m, self.resident))

    def planes_prefix(self, m):
        """The first m planes: the only code bytes a prefix-m call reads."""
        return self.planes[: packed_bytes(self.layout, m)]

    def _workspace(self, kind, n):
        # One workspace per (kind, stream), grown on demand; GEMV calls (batch <= 16) also
        # remember the size per batch, so a repeated call makes no size query.
        stream = _stream(None)
        key = (kind, stream)
        ws = self._ws.get(key)
        if kind == "gemv":
            known = self._ws.get((kind, stream, n))
            if known is not None and ws is not None and ws.numel() >= known:
                return ws
        nbytes = (gemv_workspace_bytes if kind == "gemv" else gemm_workspace_bytes)(self.layout, n)
        if ws is None or ws.numel() < nbytes:
            ws = workspace(nbytes, self.device)
            self._ws[key] = ws
        if kind == "gemv":
            self._ws[(kind, stream, n)] = nbytes
        return ws

    def decode(self, m, out=None):
        """Dense W_m [out][in] in the book dtype (bit-exact contract of aq.h)."""
        if out is None:
            out = torch.empty(self.out, self.inp, dtype=TORCH_DTYPES[DTYPES[self.book_dtype]],
                              device=self.device)
        self._check_m(m)
        aq_decode(self.layout, m, self.planes, self.books, self.scales, out)
        return out

    def gemv(self, x, m, y=None, y_dtype=None):
        """y = x W_m^T for x of shape [batch <= 16, in]."""
        xd = _dtype_code(x.dtype)
        yd = xd if y_dtype is None else y_dtype
        batch = x.shape[0]
        if y is None:
            y = torch.empty(batch, self.out, dtype=TORCH_DTYPES[yd], device=self.device)
        self._check_m(m)
        ws = self._workspace("gemv", batch)
        aq_gemv(self.layout, m, self.planes, self.books, self.scales, x, xd, batch, y, yd, ws)
        return y

    def refine(self, x, m, y_prev, y=None):
        """y = y_prev + x (s o C_{m-1}[b_{m-1}])^T: raises a prefix-(m-1) result to prefix m,
        reading plane m-1 only (y_prev None: the increment alone). y has y_prev's dtype
        (fp32 by default when y_prev is None); y may be y_prev (in place)."""
        xd = _dtype_code(x.dtype)
        batch = x.shape[0]
        yd = _dtype_code(y_prev.dtype) if y_prev is not None else AQ_F32
        if y is None:
            y = torch.empty(batch, self.out, dtype=TORCH_DTYPES[yd], device=self.device)
        self._check_m(m)
        ws = self._workspace("gemv", batch)
        aq_gemv_refine(self.layout, m, self.planes, self.books, self.scales, x, xd, batch, y_prev,
                       y, yd, ws)
        return y

    def gemm(self, x, m, y=None, y_dtype=None):
        """y = x W_m^T for x of shape [tokens, in] on the tensor cores."""
        xd = _dtype_code(x.dtype)
        yd = xd if y_dtype is None else y_dtype
        tokens = x.shape[0]
        if y is None:
            y = torch.empty(tokens, self.out, dtype=TORCH_DTYPES[yd], device=self.device)
        self._check_m(m)
        ws = self._workspace("gemm", tokens)
        aq_gemm(self.layout, m, self.planes, self.books, self.scales, x, xd, tokens, y, yd, ws)
        return y

    def wmse(self, W, H, lam=None):
        """Distortion of every prefix (Sec. 2.2 Eq. wmse-task, Sec. 5): a float64 device tensor
        d with d[k-1] = tr[(W - W^(k)) H (W - W^(k))^T] / d_out, and d[M] = sum_k lam[k-1] d[k-1]
        when lam (M weights) is given. W: [out][in] in the book dtype; H: [in][in] fp32 or
        bf16 (its symmetric part is used). All prefixes must be resident."""
        if self.resident != self.M:
            raise ValueError("the distortion needs all %d codebooks resident" % self.M)
        hd = AQ_F32 if H.dtype == torch.float32 else AQ_BF16 if H.dtype == torch.bfloat16 else None
        if hd is None:
            raise TypeError("H must be float32 or bfloat16")
        d = torch.empty(self.M + (1 if lam is not None else 0), dtype=torch.float64,
                        device=self.device)
        key = ("wmse", _stream(None))
        ws = self._ws.get(key)
        nbytes = wmse_workspace_bytes(self.layout)
        if ws is None or ws.numel() < nbytes:
            ws = workspace(nbytes, self.device)
            self._ws[key] = ws
        aq_wmse(self.layout, W, self.planes, self.books, self.scales, H, hd, lam, d, ws)
        return d

    def __call__(self, x, m):
        return self.gemv(x, m) if x.shape[0] <= 16 else self.gemm(x, m)


_group_ws = {}


def gemv_group(layers, x, m, ys=None, y_dtype=None):
    """y_l = x W_m,l^T for AQLinear layers that share the input x (aq_gemv_group: one product
    and one reduction launch at batch 1); returns the list of outputs."""
    xd = _dtype_code(x.dtype)
    yd = xd if y_dtype is None else y_dtype
    batch = x.shape[0]
    dev = layers[0].device
    for lin in layers:
        lin._check_m(m)
    if ys is None:
        ys = [torch.empty(batch, lin.out, dtype=TORCH_DTYPES[yd], device=dev) for lin in layers]
    layouts = [lin.layout for lin in layers]
    key = (tuple((lin.out, lin.inp, lin.M, lin.B) for lin in layers), batch, _stream(None), str(dev))
    ws = _group_ws.get(key)
    if ws is None:
        ws = workspace(gemv_group_workspace_bytes(layouts, batch), dev)
        _group_ws[key] = ws
    aq_gemv_group(layouts, m, [lin.planes for lin in layers], [lin.books for lin in layers],
                  [lin.scales for lin in layers], x, xd, batch, ys, yd, ws)
    return ys


def _dtype_code(dt):
    if dt == torch.float16:
        return AQ_F16
    if dt == torch.bfloat16:
        return AQ_BF16
    if dt == torch.float32:
        return AQ_F32
    raise TypeError("unsupported activation dtype %s" % dt)


def x_to_device(x_bits, x_dtype, device="cuda"):
    """Activation bit patterns (uint16, from workloads.make_x) -> device tensor of x_dtype."""
    t = _u16_to_device(x_bits, device)
    return t.view(torch.float16 if x_dtype == "f16" else torch.bfloat16)
