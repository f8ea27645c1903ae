"""CPU oracle for the additive-codebook dequantize-and-multiply (test infrastructure only).

Only the tests, the smoke check and the CPU-baseline leg of the benchmark may import this
package. It wraps oracle.cpp (ctypes, numpy arrays in and out) and shares nothing with the
CUDA library. See oracle.cpp for the paper passages each function follows.
"""
import ctypes
import os

import numpy as np

from . import build as _build

DT_F16, DT_BF16 = 0, 1
_DT = {"f16": DT_F16, "bf16": DT_BF16}

_lib = None


def lib():
    global _lib
    if _lib is None:
        # ORACLE_LIB points at another build of oracle.cpp (the mutation tests use it).
        path = os.environ.get("ORACLE_LIB") or _build.build()
        L = ctypes.CDLL(path)
        vp, i32, u16p = ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p
        L.oracle_avg_bits.restype = ctypes.c_double
        L.oracle_avg_bits.argtypes = [ctypes.c_long, ctypes.c_long, i32, i32, i32]
        L.oracle_prefix_code_bits.restype = ctypes.c_double
        L.oracle_prefix_code_bits.argtypes = [i32, i32, i32]
        L.oracle_decode.restype = i32
        L.oracle_decode.argtypes = [i32] * 6 + [vp, u16p, i32, u16p, i32, u16p]
        L.oracle_product_exact.restype = i32
        L.oracle_product_exact.argtypes = [i32] * 6 + [vp, u16p, i32, u16p, i32, u16p, i32, i32, vp]
        L.oracle_reconstruct_exact.restype = i32
        L.oracle_reconstruct_exact.argtypes = [i32] * 6 + [vp, u16p, i32, u16p, i32, vp]
        L.oracle_product_dense.restype = i32
        L.oracle_product_dense.argtypes = [i32, i32, u16p, i32, u16p, i32, i32, vp]
        L.oracle_pack.restype = i32
        L.oracle_pack.argtypes = [i32] * 5 + [vp, vp]
        L.oracle_f32_to_f16.restype = ctypes.c_uint16
        L.oracle_f32_to_f16.argtypes = [ctypes.c_float]
        L.oracle_f32_to_bf16.restype = ctypes.c_uint16
        L.oracle_f32_to_bf16.argtypes = [ctypes.c_float]
        L.oracle_f16_to_f64.restype = ctypes.c_double
        L.oracle_f16_to_f64.argtypes = [ctypes.c_uint16]
        L.oracle_bf16_to_f64.restype = ctypes.c_double
        L.oracle_bf16_to_f64.argtypes = [ctypes.c_uint16]
        L.oracle_f32_to_bits_array.restype = None
        L.oracle_f32_to_bits_array.argtypes = [vp, vp, ctypes.c_long, i32]
        L.oracle_bits_to_f64_array.restype = None
        L.oracle_bits_to_f64_array.argtypes = [vp, vp, ctypes.c_long, i32]
        L.oracle_num_threads.restype = i32
        L.oracle_num_threads.argtypes = []
        L.oracle_set_num_threads.restype = None
        L.oracle_set_num_threads.argtypes = [i32]
        _lib = L
    return _lib


def _p(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def _codes_ok(codes, B):
    want = np.uint8 if B <= 8 else np.uint16
    if codes.dtype != want or not codes.flags.c_contiguous:
        raise TypeError("codes must be C-contiguous %s for B=%d" % (np.dtype(want).name, B))


def avg_bits(d_out, d_in, g, M, B):
    """App. C, Eq. avg_bits (codes term times M)."""
    return lib().oracle_avg_bits(d_out, d_in, g, M, B)


def prefix_code_bits(g, m, B):
    return lib().oracle_prefix_code_bits(g, m, B)


def decode(layer, m):
    """Bit patterns [out][in] (uint16) of the book dtype: s[o]*sum_{k<m} C_k[b], fp32, one RNE."""
    out, inp, G, M, B = layer["out"], layer["in"], layer["G"], layer["M"], layer["B"]
    codes = layer["codes"]
    _codes_ok(codes, B)
    w = np.empty((out, inp), dtype=np.uint16)
    rc = lib().oracle_decode(out, inp, G, M, B, m, _p(codes), _p(layer["books"]),
                             _DT[layer["book_dtype"]], _p(layer["scales"]),
                             _DT[layer["scale_dtype"]], _p(w))
    if rc:
        raise ValueError("oracle_decode rejected the shape")
    return w


def product_exact(layer, x, x_dtype, m, rows=None):
    """fp64 y[t,o] = sum_i x[t,i] * (s[o]*sum_{k<m} C_k[b_{o,g,k}][e]) for t < batch.

    rows: optional (r0, r1) to evaluate only output rows r0..r1-1 (a bounded sample).
    """
    out, inp, G, M, B = layer["out"], layer["in"], layer["G"], layer["M"], layer["B"]
    codes, scales = layer["codes"], layer["scales"]
    _codes_ok(codes, B)
    if rows is not None:
        r0, r1 = rows
        codes = np.ascontiguousarray(codes[r0:r1])
        scales = np.ascontiguousarray(scales[r0:r1])
        out = r1 - r0
    x = np.ascontiguousarray(x, dtype=np.uint16).reshape(-1, inp)
    batch = x.shape[0]
    y = np.empty((batch, out), dtype=np.float64)
    rc = lib().oracle_product_exact(out, inp, G, M, B, m, _p(codes), _p(layer["books"]),
                                    _DT[layer["book_dtype"]], _p(scales),
                                    _DT[layer["scale_dtype"]], _p(x), _DT[x_dtype], batch, _p(y))
    if rc:
        raise ValueError("oracle_product_exact rejected the shape")
    return y


def reconstruct_exact(layer, m):
    """W^(m) of Sec. 5 in fp64, unrounded: [out][in], s[o]*sum_{k<m} C_k[b_{o,g,k}][e]."""
    out, inp, G, M, B = layer["out"], layer["in"], layer["G"], layer["M"], layer["B"]
    codes = layer["codes"]
    _codes_ok(codes, B)
    w = np.empty((out, inp), dtype=np.float64)
    rc = lib().oracle_reconstruct_exact(out, inp, G, M, B, m, _p(codes), _p(layer["books"]),
                                        _DT[layer["book_dtype"]], _p(layer["scales"]),
                                        _DT[layer["scale_dtype"]], _p(w))
    if rc:
        raise ValueError("oracle_reconstruct_exact rejected the shape")
    return w


def wmse(layer, W, H, ks=None):
    """Per-prefix distortion of Sec. 5 with the weighted MSE of Sec. 2.2 (Eq. wmse-task, its
    trace form): D^(k) = (1/d_out) * tr[(W - W^(k)) H (W - W^(k))^T] for k in ks (default
    1..M), W^(k) the exact prefix-k reconstruction. W: [out][in] float64 (the original weight),
    H: [in][in] float64 (the proxy X X^T / n; any square matrix is evaluated as given).
    Returns a float64 array, entry i for prefix ks[i].

    The trace is taken as the sum of the diagonal of (W - W^(k)) H (W - W^(k))^T, whose entry
    o is sum_i ((W - W^(k)) H)[o, i] * (W - W^(k))[o, i]; the out x out product itself is not
    formed. The matrix product is numpy's (fp64)."""
    out = layer["out"]
    ks = range(1, layer["M"] + 1) if ks is None else ks
    W = np.asarray(W, dtype=np.float64)
    H = np.asarray(H, dtype=np.float64)
    res = []
    for k in ks:
        E = W - reconstruct_exact(layer, k)
        res.append(float(np.sum((E @ H) * E)) / out)
    return np.array(res)


def wmse_abs(layer, W, H, ks=None):
    """(1/d_out) * sum_o |e_o| |H| |e_o|^T for each prefix (e_o = row o of W - W^(k)): the
    magnitude that first-order rounding-error bounds of D^(k) scale with."""
    out = layer["out"]
    ks = range(1, layer["M"] + 1) if ks is None else ks
    A = np.abs(np.asarray(H, dtype=np.float64))
    res = []
    for k in ks:
        E = np.abs(np.asarray(W, dtype=np.float64) - reconstruct_exact(layer, k))
        res.append(float(np.sum((E @ A) * E)) / out)
    return np.array(res)


def dbyd_loss(D, lam):
    """Sec. 5 Drop-by-Drop objective: L = sum_k lambda_k D^(k) (lam[k-1] weights prefix k)."""
    D = np.asarray(D, dtype=np.float64)
    lam = np.asarray(lam, dtype=np.float64)
    if lam.shape != D.shape:
        raise ValueError("one weight per prefix")
    total = 0.0
    for k in range(D.shape[0]):
        total += lam[k] * D[k]
    return total


def product_dense(w_bits, w_dtype, x, x_dtype):
    w_bits = np.ascontiguousarray(w_bits, dtype=np.uint16)
    out, inp = w_bits.shape
    x = np.ascontiguousarray(x, dtype=np.uint16).reshape(-1, inp)
    y = np.empty((x.shape[0], out), dtype=np.float64)
    rc = lib().oracle_product_dense(out, inp, _p(w_bits), _DT[w_dtype], _p(x), _DT[x_dtype],
                                    x.shape[0], _p(y))
    if rc:
        raise ValueError("oracle_product_dense rejected the shape")
    return y


def pack(layer):
    """Packed code planes (see oracle.cpp for the index map) as a flat uint8 array."""
    out, inp, G, M, B = layer["out"], layer["in"], layer["G"], layer["M"], layer["B"]
    codes = layer["codes"]
    _codes_ok(codes, B)
    rows_pad = (out + 31) // 32 * 32
    ng_pad = (inp // G + 31) // 32 * 32
    nbytes = M * rows_pad * ng_pad * (1 if B <= 8 else 2) // (2 if B <= 4 else 1)
    buf = np.zeros(nbytes, dtype=np.uint8)
    rc = lib().oracle_pack(out, inp, G, M, B, _p(codes), _p(buf))
    if rc:
        raise ValueError("oracle_pack rejected the shape")
    return buf


def f32_to_f16(v):
    return lib().oracle_f32_to_f16(float(v))


def f32_to_bf16(v):
    return lib().oracle_f32_to_bf16(float(v))


def f16_to_f64(h):
    return lib().oracle_f16_to_f64(int(h))


def bf16_to_f64(b):
    return lib().oracle_bf16_to_f64(int(b))


def round_bits(a, dtype):
    """float32 array -> fp16/bf16 bit patterns with the oracle's own round-to-nearest-even."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    out = np.empty(a.shape, dtype=np.uint16)
    lib().oracle_f32_to_bits_array(_p(a), _p(out), a.size, _DT[dtype])
    return out


def bits_value(v, dtype):
    """fp16/bf16 bit patterns -> float64 values with the oracle's own widening."""
    v = np.ascontiguousarray(v, dtype=np.uint16)
    out = np.empty(v.shape, dtype=np.float64)
    lib().oracle_bits_to_f64_array(_p(v), _p(out), v.size, _DT[dtype])
    return out


def num_threads():
    return lib().oracle_num_threads()


def set_num_threads(n):
    """Threads the oracle's OpenMP loops use from now on (timing only; results do not depend
    on it)."""
    lib().oracle_set_num_threads(int(n))


def widen(bits, dtype):
    """Exact widening of fp16/bf16 bit patterns to float64 (numpy, vectorised)."""
    bits = np.asarray(bits, dtype=np.uint16)
    if dtype == "f16":
        return bits.view(np.float16).astype(np.float64)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def beam_update(layer, W, H, lam, K, only=None):
    """One code update of Alg. 1 ("update assignments b using beam search"; App. C describes
    it as a search for the codeword combinations that minimise the error of the layer's
    outputs), in this reading: for every row o and group g, with the codes of the row's other
    groups held at their current values, the group's M codes are chosen by a beam search of
    width K over the books in order 0..M-1 that minimises the Drop-by-Drop objective of Sec. 5
    restricted to the row, sum_k lam[k-1] * e^(k) S e^(k)^T with e^(k) = W[o] - W^(k)[o] and
    S = (H + H^T)/2 (only the symmetric part of H enters a trace form). Every group is updated
    from the same current codes. Changing group g moves only its block of e^(k), by
    delta_k = w_g - s_o * (sum_{j<k} C_j[b_j]), so the terms that depend on the group's codes
    are delta_k^T S_gg delta_k + 2 delta_k^T h_k with h_k the cross term of the block with the
    rest of the row, h_k = (S e^(k))_g - S_gg e^(k)_g.

    Beam: states (codes chosen so far, their codeword sum P, score); from the single empty
    state, book t extends every state by every codeword c of C_t, scoring
    score + lam[t] * (d^T S_gg d + 2 d^T h_{t+1}) with d = w_g - s_o (P + C_t[c]); the K best
    extensions are kept, ordered by (score, rank of the parent state, c). The result is the
    first state after book M-1. Scores in fp64.

    W: [out][in] float64, H: [in][in] float64, lam: M weights, K >= 1. only: optional
    iterable of (o, g) pairs; the other groups keep their codes. Returns new codes with the
    shape and dtype of layer["codes"]."""
    out, inp, G, M, B = layer["out"], layer["in"], layer["G"], layer["M"], layer["B"]
    codes = np.asarray(layer["codes"])
    books = widen(layer["books"], layer["book_dtype"]).reshape(M, 1 << B, G)
    s = widen(layer["scales"], layer["scale_dtype"])
    W = np.asarray(W, dtype=np.float64)
    H = np.asarray(H, dtype=np.float64)
    S = (H + H.T) / 2
    lam = np.asarray(lam, dtype=np.float64)
    E = [W - reconstruct_exact(layer, k) for k in range(1, M + 1)]   # e^(k), k = 1..M
    V = [e @ S for e in E]                                          # rows of S e^(k)
    new = codes.copy()
    nb = 1 << B
    pairs = [(o, g) for o in range(out) for g in range(inp // G)] if only is None else only
    for o, g in pairs:
        blk = slice(g * G, (g + 1) * G)
        Sgg = S[blk, blk]
        wg = W[o, blk]
        h = [V[k][o, blk] - Sgg @ E[k][o, blk] for k in range(M)]
        states = [((), np.zeros(G), 0.0)]
        for t in range(M):
            score, rank, cw = [], [], []
            for r, (cs, P, sc) in enumerate(states):
                D = wg - s[o] * (P + books[t])          # row c: d for codeword c of C_t
                q = np.einsum("ce,ef,cf->c", D, Sgg, D)
                score.append(sc + lam[t] * (q + 2.0 * (D @ h[t])))
                rank.append(np.full(nb, r))
                cw.append(np.arange(nb))
            score, rank, cw = np.concatenate(score), np.concatenate(rank), np.concatenate(cw)
            keep = np.lexsort((cw, rank, score))[:K]    # by score, then parent rank, then c
            states = [(states[rank[i]][0] + (int(cw[i]),), states[rank[i]][1] + books[t, cw[i]],
                       float(score[i])) for i in keep]
        new[o, g, :] = states[0][0]
    return new


def row_objective(layer, W, H, lam, o):
    """sum_k lam[k-1] * e^(k) S e^(k)^T for row o (S = (H + H^T)/2, e^(k) = W[o] - W^(k)[o],
    exact reconstruction): the quantity the code update minimises, evaluated directly."""
    M = layer["M"]
    W = np.asarray(W, dtype=np.float64)
    H = np.asarray(H, dtype=np.float64)
    S = (H + H.T) / 2
    tot = 0.0
    for k in range(1, M + 1):
        e = W[o] - reconstruct_exact(layer, k)[o]
        tot += lam[k - 1] * float(e @ S @ e)
    return tot
