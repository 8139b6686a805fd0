"""Seeded synthetic calibration activations X~ [tokens][din] in float16.

Input generation only (no part of the method's arithmetic): the rows stand
in for a layer's inputs over the calibration set (Sec. 3.1: X~ stacks the
inputs a layer receives with the quantized preceding layers; the paper
calibrates on 128 sequences of 2048 tokens, Sec. 4.1 / App. B).  The recipe
matches the Hessian generator of ``layers.py``: a rank-r correlated part, an
independent part with per-channel variance in [D_lo, 1] and a few outlier
channels scaled by ``out_scale``, which gives the heavy-diagonal, low-rank
structure of real calibration Hessians.  Values are rounded once to float16,
the precision in which the paper holds activations.
"""
from __future__ import annotations

import math

import numpy as np

# name -> din, tokens, rank of the correlated part, outlier channels, seed
ACT_CONFIGS = {
    # input of q/k/v/gate/up of a Llama-2-7B block, 128 x 2048 tokens
    "llama2_7b_attn_in_4096_n262144": dict(din=4096, tokens=262144, rank=64, n_out=16,
                                           out_scale=30.0, D_lo=0.05, seed=60),
    # input of down_proj (the MLP width), 64 x 2048 tokens
    "llama2_7b_down_in_11008_n131072": dict(din=11008, tokens=131072, rank=64, n_out=32,
                                            out_scale=30.0, D_lo=0.05, seed=61),
}


def activations_np(tokens, din, rank=8, n_out=2, out_scale=30.0, D_lo=0.05, seed=0):
    """float16 [tokens][din] drawn with NumPy's PCG64 (small cases)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    L = rng.standard_normal((din, rank)) * (2.0 / math.sqrt(rank))
    D = rng.uniform(D_lo, 1.0, din)
    col = np.ones(din)
    if n_out:
        col[rng.choice(din, n_out, replace=False)] = out_scale
    U = rng.standard_normal((tokens, rank))
    E = rng.standard_normal((tokens, din))
    X = (U @ L.T + E * np.sqrt(D)) * col
    return X.astype(np.float16)


def integer_activations_np(tokens, din, amax=8, seed=0):
    """float16 [tokens][din] holding integers in [-amax, amax]: every product
    and, while tokens * amax^2 < 2^24, every sum over tokens is exact in
    float32, so a float32 accumulation must reproduce X^T X bit for bit."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.integers(-amax, amax + 1, size=(tokens, din)).astype(np.float16)


def activations_torch(tokens, din, rank, n_out, out_scale, D_lo, seed, device, chunk=16384):
    """The same recipe drawn with ``torch.Generator`` on ``device`` (full-size
    cases), generated chunk by chunk into one float16 [tokens][din] tensor."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    L = torch.randn(din, rank, generator=gen, device=device) * (2.0 / math.sqrt(rank))
    D = torch.rand(din, generator=gen, device=device) * (1.0 - D_lo) + D_lo
    col = torch.ones(din, device=device)
    if n_out:
        idx = torch.randperm(din, generator=gen, device=device)[:n_out]
        col[idx] = out_scale
    sqD = D.sqrt()
    X = torch.empty(tokens, din, dtype=torch.float16, device=device)
    done = 0
    while done < tokens:
        m = min(chunk, tokens - done)
        U = torch.randn(m, rank, generator=gen, device=device)
        E = torch.randn(m, din, generator=gen, device=device)
        X[done:done + m] = ((U @ L.T + E * sqD) * col).half()
        done += m
    return X


def config_activations(name, device="cuda", tokens=None):
    """One named activation workload on ``device`` (``tokens`` overrides n)."""
    c = ACT_CONFIGS[name]
    return activations_torch(tokens or c["tokens"], c["din"], c["rank"], c["n_out"],
                             c["out_scale"], c["D_lo"], c["seed"], device)
