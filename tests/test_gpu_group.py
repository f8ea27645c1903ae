"""The GEMV of a group of layers that share the activations (aq_gemv_group: the query/key/value
or gate/up projections of a decoder block; the product y = x W_m^T of Sec. 2.2 with the prefix
reconstruction of Sec. 3.2 / Sec. 5 for each layer). At batch 1 the layers' products run as one
kernel and their reductions as one kernel; every layer's partial sums and their summation
order are those of its own call, so each output must equal the same layer's aq_gemv output
bit for bit, and the oracle within the product tolerance. Covered: ragged rows and slices,
every prefix, both activation types, a group one launch cannot serve (a layer too small to
keep every CTA within two layers: the layers then run one after the other), other batches
(one call per layer), layers whose weights are not marked static, and the Llama-3-8B
projections."""
import numpy as np
import pytest
import torch

import aq_testutil as U
import oracle
import paper_2606_12876_gb300 as aq
import workloads
from paper_2606_12876_gb300.linear import AQLinear, gemv_group, x_to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def gpu():
    U.require_gpu()


def _layers(shapes, inp, M, bdt="f16", seed=0):
    return [workloads.make_layer(out, inp, G=8, M=M, B=8, book_dtype=bdt, book_std=0.05,
                                 scale_dtype="f16", seed=seed + i) for i, out in enumerate(shapes)]


def _check_group(layers, x_bits, xdt, ms, batch=1, static=True, oracle_check=True):
    lins = [AQLinear.from_layer(l) for l in layers]
    if not static:
        lins[-1].layout.flags = 0
    x = x_to_device(x_bits[:batch], xdt)
    for m in ms:
        ys = gemv_group(lins, x, m, y_dtype=aq.AQ_F32)
        for l, (lin, layer, y) in enumerate(zip(lins, layers, ys)):
            single = lin.gemv(x, m, y_dtype=aq.AQ_F32)
            assert torch.equal(y, single), "layer %d m=%d: group and single call differ" % (l, m)
            if oracle_check:
                U.assert_product_close(U.to_f64(y), oracle.product_exact(layer, x_bits[:batch], xdt, m),
                                       "layer %d m=%d" % (l, m))


@pytest.mark.parametrize("xdt", ["f16", "bf16"])
def test_group_ragged_every_prefix(xdt):
    """Three layers of 300, 96 and 200 rows over 1032 inputs (5 slices, the last with one
    group), four books: one product launch and one reduction per call."""
    layers = _layers((300, 96, 200), 1032, 4, seed=3)
    x_bits = workloads.make_x(1, 1032, xdt, seed=4)
    _check_group(layers, x_bits, xdt, (1, 2, 3, 4))


def test_group_two_layers_bf16_books():
    layers = _layers((640, 520), 2056, 3, bdt="bf16", seed=5)
    x_bits = workloads.make_x(1, 2056, "bf16", seed=6)
    _check_group(layers, x_bits, "bf16", (1, 3))


def test_group_falls_back_when_a_layer_is_too_small():
    """A 32-row middle layer (5 items at m = 1) between two 4096-row ones: a CTA's items would
    span three layers, so the layers run as separate calls, with the same results."""
    layers = _layers((4096, 32, 4096), 1280, 2, seed=7)
    x_bits = workloads.make_x(1, 1280, "f16", seed=8)
    _check_group(layers, x_bits, "f16", (1, 2))


@pytest.mark.parametrize("batch", [2, 5, 16])
def test_group_other_batches(batch):
    layers = _layers((300, 96), 1032, 4, seed=9)
    x_bits = workloads.make_x(16, 1032, "f16", seed=10)
    _check_group(layers, x_bits, "f16", (1, 4), batch=batch)


def test_group_with_weights_not_static():
    """One layer without AQ_LAYOUT_STATIC_WEIGHTS: the group requests nothing before the grid
    wait; results unchanged."""
    layers = _layers((300, 96, 200), 1032, 4, seed=11)
    x_bits = workloads.make_x(1, 1032, "f16", seed=12)
    _check_group(layers, x_bits, "f16", (2, 4), static=False)


def test_group_llama8b_projections():
    """q/k/v (4096, 1024, 1024 rows) and gate/up (14336 rows twice) of the Llama-3-8B block,
    bf16 activations: bit-identical to the single calls at every prefix."""
    blk = dict(workloads.config_layers("llama8b_block"))
    x_bits = workloads.config_x("llama8b_block", 1, 4096)
    for names in (("q_proj", "k_proj", "v_proj"), ("gate_proj", "up_proj")):
        _check_group([blk[n] for n in names], x_bits, "bf16", (1, 2, 3, 4), oracle_check=False)
