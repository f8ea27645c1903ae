"""Seeded synthetic inputs for the additive-codebook layers (shared by the oracle and the GPU path).

This module holds NONE of the method's arithmetic: it only draws random numbers and rounds
them to storage formats. The shapes and value distributions stand in for the paper's
workloads (Llama-3-8B / Llama-2-70B linear-layer shapes, g = 8, 8-bit codes, M <= 5 books,
Gaussian-looking weights), which need model weights and datasets that are not available.

Draw order per layer (one numpy PCG64 stream per layer): books, codes, scales. Activations
come from their own stream. All values are returned as numpy arrays of raw bit patterns
(uint16 for fp16/bf16) or code integers (uint8 for B = 8, uint16 for B = 16).
"""
import numpy as np
import torch

# name -> workload description. "layers" lists (name, out_features, in_features).
CONFIGS = {
    "single_1024": dict(
        layers=[("linear", 1024, 1024)], G=8, M=2, B=8, book_dtype="f16", book_std=0.02,
        scale_dtype="f16", x_dtype="f16", batches=(1,), ms=(1, 2), seed=0),
    "attn_4096": dict(
        layers=[("attn_proj", 4096, 4096)], G=8, M=4, B=8, book_dtype="f16", book_std=0.02,
        scale_dtype="f16", x_dtype="f16", batches=(1, 4, 16), ms=(1, 2, 3, 4), seed=1),
    "llama8b_block": dict(
        layers=[("q_proj", 4096, 4096), ("k_proj", 1024, 4096), ("v_proj", 1024, 4096),
                ("o_proj", 4096, 4096), ("gate_proj", 14336, 4096), ("up_proj", 14336, 4096),
                ("down_proj", 4096, 14336)],
        G=8, M=4, B=8, book_dtype="f16", book_std=0.02, scale_dtype="f16", x_dtype="bf16",
        batches=(1, 8), ms=(1, 2, 3, 4), seed=2),
    "big_book_8192": dict(
        layers=[("linear", 8192, 8192)], G=8, M=2, B=16, book_dtype="f16", book_std=0.02,
        scale_dtype="f16", x_dtype="f16", batches=(1, 16), ms=(1, 2), seed=3),
    "llama70b_up_prefill": dict(
        layers=[("up_proj", 28672, 8192)], G=8, M=4, B=8, book_dtype="bf16", book_std=0.015,
        scale_dtype="bf16", x_dtype="bf16", batches=(4096,), ms=(1, 2, 3, 4), seed=4),
}


def to_bits(a, dtype):
    """Round float32 values to fp16/bf16 (round-to-nearest-even) and return the bit patterns."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    if dtype == "f16":
        return a.astype(np.float16).view(np.uint16)
    if dtype == "bf16":
        t = torch.from_numpy(a).to(torch.bfloat16)
        return t.view(torch.int16).numpy().view(np.uint16).copy()
    raise ValueError(dtype)


def make_layer(out, inp, G=8, M=4, B=8, book_dtype="f16", book_std=0.02, scale_dtype="f16",
               seed=0, scale_lo=0.5, scale_hi=1.5):
    """One quantized linear layer: books [M][2^B][G], codes (out, in/G, M), scales [out]."""
    if inp % G:
        raise ValueError("in_features must be a multiple of G")
    rng = np.random.Generator(np.random.PCG64(seed))
    nb = 1 << B
    books = to_bits(rng.standard_normal((M, nb, G), dtype=np.float32) * np.float32(book_std),
                    book_dtype)
    cdt = np.uint8 if B <= 8 else np.uint16
    codes = rng.integers(0, nb, size=(out, inp // G, M), dtype=cdt)
    scales = to_bits(rng.uniform(scale_lo, scale_hi, size=out).astype(np.float32), scale_dtype)
    return dict(out=out, **{"in": inp}, G=G, M=M, B=B, books=books, codes=codes, scales=scales,
                book_dtype=book_dtype, scale_dtype=scale_dtype)


def make_x(batch, inp, x_dtype="f16", seed=0):
    """Activations [batch][in] drawn N(0, 1), rounded to x_dtype."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return to_bits(rng.standard_normal((batch, inp), dtype=np.float32), x_dtype)


def layer_seed(seed, idx):
    """Seed of the idx-th layer of a workload (independent stream per layer)."""
    return int(np.random.SeedSequence([seed, idx]).generate_state(1)[0])


def x_seed(seed, batch):
    return int(np.random.SeedSequence([seed, 1000 + batch]).generate_state(1)[0])


def config_layers(name, only=None):
    """Yield (layer_name, layer_dict) for a named workload."""
    cfg = CONFIGS[name]
    for idx, (lname, out, inp) in enumerate(cfg["layers"]):
        if only is not None and lname not in only:
            continue
        yield lname, make_layer(out, inp, cfg["G"], cfg["M"], cfg["B"], cfg["book_dtype"],
                                cfg["book_std"], cfg["scale_dtype"], layer_seed(cfg["seed"], idx))


def config_x(name, batch, inp):
    cfg = CONFIGS[name]
    return make_x(batch, inp, cfg["x_dtype"], x_seed(cfg["seed"], batch) + inp)
