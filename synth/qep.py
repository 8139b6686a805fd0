"""Seeded inputs for the propagation-corrected (mu) target.

Input generation only (none of the method's arithmetic).  App.
"Propagation-Corrected Targets and QEP" mixes the layer's full-precision
inputs X with the inputs X~ it receives after the quantized preceding
layers.  Here X~ is drawn with the activation recipe of ``activations.py``
and X = X~ + drift, the drift being a small correlated perturbation (the
error the quantized preceding layers leave), both rounded to float16.  The
three Gram matrices the mu-target needs are formed from those float16 values
in float64 and rounded once to float32, normalised by the token count like
the Hessians of ``layers.py``:

    H  = X~^T X~ / n + nu2 I,   K = X~^T X / n,   XX = X^T X / n,

with nu2 = damp * mean(diag(X~^T X~ / n)).  Weights and the RTN host state
come from ``layers.py``.
"""
from __future__ import annotations

import dataclasses

import numpy as np

from .activations import activations_np
from .layers import rtn_host_np, weights_np


@dataclasses.dataclass
class MuLayer:
    """A layer with the inputs of the mu-target: float32 W [dout][din],
    H, K, XX [din][din], the RTN host state and nu2 (float)."""

    name: str
    W: np.ndarray
    H: np.ndarray
    K: np.ndarray
    XX: np.ndarray
    nu2: float
    S0: np.ndarray
    Q0: np.ndarray
    Z: np.ndarray
    bits: int
    g: int
    K_iters: int
    Xq: np.ndarray = None        # float16 X~ [n][din]
    Xf: np.ndarray = None        # float16 X  [n][din]


def drifted_activations_np(tokens, din, drift=0.05, rank=8, n_out=2, seed=0):
    """(X~, X) as float16 [tokens][din]: X = X~ + drift * (a rank-4 mix of X~'s
    channels + independent noise), scaled to the per-channel spread of X~."""
    Xq = activations_np(tokens, din, rank=rank, n_out=n_out, seed=seed)
    rng = np.random.Generator(np.random.PCG64(seed + 7919))
    X64 = Xq.astype(np.float64)
    sd = X64.std(axis=0) + 1e-3
    M = rng.standard_normal((din, 4)) @ rng.standard_normal((4, din)) / (2.0 * np.sqrt(din))
    E = (X64 / sd) @ M + 0.5 * rng.standard_normal((tokens, din))
    Xf = (X64 + drift * E * sd).astype(np.float16)
    return Xq, Xf


def mu_layer(din, dout, g, bits, K_iters=3, tokens=None, drift=0.05, damp=0.01, seed=0,
             w_std=0.02, keep_activations=True):
    """A small seeded mu-target layer (NumPy, PCG64)."""
    tokens = tokens if tokens is not None else 8 * din
    Xq, Xf = drifted_activations_np(tokens, din, drift=drift, rank=max(1, din // 32),
                                    seed=seed)
    A = Xq.astype(np.float64)
    B = Xf.astype(np.float64)
    H0 = A.T @ A / tokens
    nu2 = float(np.float32(damp * np.mean(np.diag(H0))))
    H = (H0 + nu2 * np.eye(din)).astype(np.float32)
    K = (A.T @ B / tokens).astype(np.float32)
    XX = (B.T @ B / tokens).astype(np.float32)
    rng = np.random.Generator(np.random.PCG64(seed + 104729))
    W = weights_np(rng, dout, din, w_std, 0.005, 8.0)
    S0, Q0, Z = rtn_host_np(W, bits, g)
    return MuLayer(f"mu_{dout}x{din}_g{g}_w{bits}_s{seed}", W, H, K, XX, nu2, S0, Q0, Z, bits,
                   g, K_iters, Xq if keep_activations else None, Xf if keep_activations else None)


def mu_grams_torch(din, tokens, rank, n_out, out_scale, D_lo, seed, device, drift=0.05,
                   damp=0.01, chunk=8192):
    """Full-size (H, K, XX, nu2) on ``device``: X~ drawn chunk by chunk with the
    activation recipe and X = X~ + drift (a rank-4 channel mix of X~ plus
    noise, scaled per channel), both rounded to float16; each chunk's
    products formed in float32 (no TF32) and summed in float64; normalised
    by the token count; returned as float32 matrices."""
    import math

    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    L = torch.randn(din, rank, generator=gen, device=device) * (2.0 / math.sqrt(rank))
    D = torch.rand(din, generator=gen, device=device) * (1.0 - D_lo) + D_lo
    col = torch.ones(din, device=device)
    if n_out:
        idx = torch.randperm(din, generator=gen, device=device)[:n_out]
        col[idx] = out_scale
    sd = torch.sqrt((L * L).sum(1) + D) * col          # per-channel spread of X~
    M = (torch.randn(din, 4, generator=gen, device=device)
         @ torch.randn(4, din, generator=gen, device=device)) / (2.0 * math.sqrt(din))
    sqD = D.sqrt()
    H0 = torch.zeros(din, din, dtype=torch.float64, device=device)
    K = torch.zeros_like(H0)
    XX = torch.zeros_like(H0)
    prev = torch.get_float32_matmul_precision()
    torch.set_float32_matmul_precision("highest")
    try:
        done = 0
        while done < tokens:
            m = min(chunk, tokens - done)
            U = torch.randn(m, rank, generator=gen, device=device)
            E = torch.randn(m, din, generator=gen, device=device)
            Xq = ((U @ L.T + E * sqD) * col).half().float()
            N = torch.randn(m, din, generator=gen, device=device)
            Xf = (Xq + drift * ((Xq / sd) @ M + 0.5 * N) * sd).half().float()
            H0 += (Xq.T @ Xq).double()
            K += (Xq.T @ Xf).double()
            XX += (Xf.T @ Xf).double()
            done += m
    finally:
        torch.set_float32_matmul_precision(prev)
    H0 /= tokens
    K /= tokens
    XX /= tokens
    nu2 = float(torch.tensor(damp * H0.diagonal().mean().item()).float())
    H = H0 + nu2 * torch.eye(din, dtype=torch.float64, device=device)
    return H.float(), K.float(), XX.float(), nu2


def mu_config_layer(name, device="cuda", drift=0.05):
    """A named full-size layer of ``layers.CONFIGS`` with mu-target inputs:
    (Layer, K, XX, nu2); the Layer's H is X~^T X~ / n + nu2 I."""
    from .layers import CONFIGS, config_layer
    c = CONFIGS[name]
    H, K, XX, nu2 = mu_grams_torch(c["din"], c["tokens"], c["rank"], c["n_out"], c["out_scale"],
                                   c["D_lo"], 500 + c["seed"], device, drift=drift)
    return config_layer(name, device=device, H=H), K, XX, nu2
