"""Helpers shared by the test files (tolerances, building the library, device transfers)."""
import os

import numpy as np
import pytest
import torch

# Product tolerance (stated for the dequantize-and-multiply path): relative Frobenius error
# <= 2e-3 and, per element, |y - y_ref| <= 1e-2 * (1 + |y_ref|), against the oracle's fp64
# product of the exactly widened stored values.
REL_FRO = 2e-3
ELEM_ABS = 1e-2


def ensure_built():
    import paper_2606_12876_gb300.build as b
    b.build()


def has_gpu():
    return torch.cuda.is_available()


def require_gpu():
    if not has_gpu():
        pytest.skip("needs a CUDA GPU")
    ensure_built()


def product_errors(y, y_ref):
    y = np.asarray(y, dtype=np.float64)
    y_ref = np.asarray(y_ref, dtype=np.float64)
    diff = y - y_ref
    denom = np.linalg.norm(y_ref)
    rel = np.linalg.norm(diff) / denom if denom > 0 else np.linalg.norm(diff)
    elem = np.max(np.abs(diff) / (1.0 + np.abs(y_ref))) if diff.size else 0.0
    return rel, elem


def assert_product_close(y, y_ref, what=""):
    rel, elem = product_errors(y, y_ref)
    assert rel <= REL_FRO, "%s: relative Frobenius error %.3e > %.0e" % (what, rel, REL_FRO)
    assert elem <= ELEM_ABS, "%s: per-element error %.3e > %.0e" % (what, elem, ELEM_ABS)
    return rel, elem


def to_f64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def bits_of(t):
    """Raw 16-bit patterns of an fp16/bf16 device tensor, as numpy uint16."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
