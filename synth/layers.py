"""Seeded synthetic layers shaped like the paper's workloads.

This module is the only code that both the CUDA path's tests and the oracle
use.  It holds none of JARQ's arithmetic: it draws weights and calibration
activations, accumulates the Hessian ``H = X^T X / n + damping * I`` and runs
the round-to-nearest (RTN) host quantizer that supplies the initial state
``(S0, Q0, Z)``.

Shapes stand in for the paper's Llama-2-7B / Llama-3-8B linear layers at
W3A16 / W4A16, group size 128, calibrated on 128 x 2048 tokens (Sec. 4.1
"Setup"; App. B "Calibration and Host Quantizers").  No dataset or model
weights are used: activations are drawn from ``N(0, L L^T + diag(D))`` with
a few outlier channels, which reproduces the low-rank, correlated, heavy
diagonal structure of real calibration Hessians.

Small layers (the tiny 256x256 case and test cases) are drawn with NumPy's
PCG64 on the host.  Full-size layers are drawn with ``torch.Generator`` on
the device they are requested on (the calibration product is 9-64 TFLOP);
both the oracle and the CUDA path then read the same tensors.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np


@dataclasses.dataclass
class Layer:
    """One synthetic layer with its RTN host state.

    ``W``: float32 [dout][din]; ``H``: float32 [din][din];
    ``S0``: float32 [dout][G]; ``Q0``: uint8 [dout][din];
    ``Z``: int32 [dout][G].  Arrays are numpy arrays or torch tensors.
    """

    name: str
    W: object
    H: object
    S0: object
    Q0: object
    Z: object
    bits: int
    g: int
    K: int

    @property
    def din(self):
        return int(self.W.shape[1])

    @property
    def dout(self):
        return int(self.W.shape[0])

    @property
    def G(self):
        return self.din // self.g


# Workload table: name -> (din, dout, g, bits, K, rank of L, outlier channels,
# tokens, weight law, RTN clip ratio, seed).
CONFIGS = {
    "tiny_256x256_g64_w3": dict(din=256, dout=256, g=64, bits=3, K=5, rank=16,
                                n_out=4, out_scale=20.0, tokens=2048,
                                w_std=0.02, w_out_frac=0.005, w_out_mul=8.0,
                                law="normal", clip=1.0, D_lo=0.1, seed=0),
    "llama2_7b_q_proj_4096x4096_g128_w3": dict(
        din=4096, dout=4096, g=128, bits=3, K=10, rank=64, n_out=16,
        out_scale=30.0, tokens=262144, w_std=0.015, w_out_frac=0.001,
        w_out_mul=10.0, law="normal", clip=1.0, D_lo=0.05, seed=2),
    # the q_proj layer at group size 64 (App. "Group size"): 64 groups per row
    "llama2_7b_q_proj_4096x4096_g64_w3": dict(
        din=4096, dout=4096, g=64, bits=3, K=10, rank=64, n_out=16,
        out_scale=30.0, tokens=262144, w_std=0.015, w_out_frac=0.001,
        w_out_mul=10.0, law="normal", clip=1.0, D_lo=0.05, seed=2),
    "llama2_7b_down_proj_4096x11008_g128_w4": dict(
        din=11008, dout=4096, g=128, bits=4, K=10, rank=64, n_out=32,
        out_scale=30.0, tokens=131072, w_std=0.015, w_out_frac=0.001,
        w_out_mul=10.0, law="normal", clip=0.9, D_lo=0.05, seed=3),
    "llama3_8b_gate_proj_14336x4096_g128_w3": dict(
        din=4096, dout=14336, g=128, bits=3, K=10, rank=64, n_out=16,
        out_scale=30.0, tokens=262144, w_std=0.015, w_out_frac=0.001,
        w_out_mul=10.0, law="student_t4", clip=1.0, D_lo=0.05, seed=4),
}

# The Llama-2-7B decoder block: (layer, dout, din, Hessian it reads).
BLOCK_LLAMA2_7B = [
    ("q_proj", 4096, 4096, "attn_in"), ("k_proj", 4096, 4096, "attn_in"),
    ("v_proj", 4096, 4096, "attn_in"), ("o_proj", 4096, 4096, "o_in"),
    ("gate_proj", 11008, 4096, "attn_in"), ("up_proj", 11008, 4096, "attn_in"),
    ("down_proj", 4096, 11008, "down_in"),
]
BLOCK_HESSIANS = {"attn_in": (4096, 50), "o_in": (4096, 51), "down_in": (11008, 52)}


# --------------------------------------------------------------------------
# RTN host (App. B: "RTN rounds weights to the quantization grid")
# --------------------------------------------------------------------------

def rtn_host_np(W, bits, g, clip=1.0):
    """Asymmetric min-max round-to-nearest per group (NumPy, float64).

    ``s = clip*(max - min)/qmax`` (1 where zero), ``z = clamp(rint(-clip*min/s))``,
    ``q = clamp(rint(w/s) + z)``.  Returns float32 scales, uint8 codes and
    int32 zero points.
    """
    W = np.asarray(W, dtype=np.float64)
    p, d = W.shape
    qmax = (1 << bits) - 1
    Wg = W.reshape(p, d // g, g)
    lo = Wg.min(axis=2) * clip
    hi = Wg.max(axis=2) * clip
    s = (hi - lo) / qmax
    s = np.where(s == 0, 1.0, s).astype(np.float32).astype(np.float64)
    z = np.clip(np.rint(-lo / s), 0, qmax)
    q = np.clip(np.rint(Wg / s[..., None]) + z[..., None], 0, qmax)
    return (s.astype(np.float32), q.reshape(p, d).astype(np.uint8),
            z.astype(np.int32))


def rtn_host_torch(W, bits, g, clip=1.0):
    """The same RTN host on torch tensors (any device)."""
    import torch
    W64 = W.double()
    p, d = W64.shape
    qmax = (1 << bits) - 1
    Wg = W64.view(p, d // g, g)
    lo = Wg.amin(dim=2) * clip
    hi = Wg.amax(dim=2) * clip
    s = (hi - lo) / qmax
    s = torch.where(s == 0, torch.ones_like(s), s).float().double()
    z = torch.clamp(torch.round(-lo / s), 0, qmax)
    q = torch.clamp(torch.round(Wg / s[..., None]) + z[..., None], 0, qmax)
    return s.float(), q.reshape(p, d).to(torch.uint8), z.to(torch.int32)


# --------------------------------------------------------------------------
# NumPy generators (small layers)
# --------------------------------------------------------------------------

def hessian_np(rng, din, rank, n_out, out_scale, tokens, D_lo, damp=0.01):
    """``H = X^T X / n + damp * mean(diag) * I`` from correlated activations."""
    L = rng.standard_normal((din, rank))
    D = rng.uniform(D_lo, 1.0, din)
    U = rng.standard_normal((tokens, rank))
    E = rng.standard_normal((tokens, din))
    X = U @ L.T + E * np.sqrt(D)
    if n_out:
        X[:, rng.choice(din, n_out, replace=False)] *= out_scale
    X = X.astype(np.float32).astype(np.float64)
    H = X.T @ X / tokens
    H += damp * np.mean(np.diag(H)) * np.eye(din)
    return H.astype(np.float32), X.astype(np.float32)


def weights_np(rng, dout, din, w_std, w_out_frac, w_out_mul, law="normal"):
    if law == "student_t4":
        t = rng.standard_t(4, (dout, din))
        W = t * (w_std / math.sqrt(2.0))
    else:
        W = rng.normal(0.0, w_std, (dout, din))
    mask = rng.random((dout, din)) < w_out_frac
    W[mask] *= w_out_mul
    return W.astype(np.float32)


def small_layer(din, dout, g, bits, K=3, seed=0, rank=None, tokens=None,
                n_out=2, out_scale=20.0, w_std=0.02, w_out_frac=0.005,
                w_out_mul=8.0, D_lo=0.1, clip=1.0, law="normal",
                return_X=False, name=None):
    """A small seeded layer (NumPy, PCG64) with the tiny-layer recipe."""
    rng = np.random.Generator(np.random.PCG64(seed))
    rank = rank if rank is not None else max(1, din // 16)
    tokens = tokens if tokens is not None else 8 * din
    W = weights_np(rng, dout, din, w_std, w_out_frac, w_out_mul, law)
    H, X = hessian_np(rng, din, rank, n_out, out_scale, tokens, D_lo)
    S0, Q0, Z = rtn_host_np(W, bits, g, clip)
    lay = Layer(name or f"small_{dout}x{din}_g{g}_w{bits}_s{seed}", W, H, S0, Q0, Z, bits, g, K)
    return (lay, X) if return_X else lay


def tiny_layer(return_X=False):
    """The tiny 256x256, g=64, 3-bit layer (seed 0, 2048 tokens, K=5)."""
    c = CONFIGS["tiny_256x256_g64_w3"]
    return small_layer(c["din"], c["dout"], c["g"], c["bits"], K=c["K"], seed=c["seed"],
                       rank=c["rank"], tokens=c["tokens"], n_out=c["n_out"],
                       out_scale=c["out_scale"], w_std=c["w_std"],
                       w_out_frac=c["w_out_frac"], w_out_mul=c["w_out_mul"],
                       D_lo=c["D_lo"], clip=c["clip"], law=c["law"],
                       return_X=return_X, name="tiny_256x256_g64_w3")


# --------------------------------------------------------------------------
# torch generators (full-size layers, built on the requested device)
# --------------------------------------------------------------------------

def hessian_torch(din, rank, n_out, out_scale, tokens, D_lo, seed, device,
                  chunk=8192, damp=0.01, token_seed=None):
    """``X^T X / n + damp*mean(diag)*I`` accumulated chunk by chunk.

    Each 8192-token chunk's product is formed in float32 (full-precision
    matmul, no TF32) and summed in float64.  With ``token_seed`` the
    distribution (L, D, outlier channels) is the one of ``seed`` and the
    tokens are drawn from ``token_seed``: a held-out calibration set.
    """
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    L = torch.randn(din, rank, generator=gen, device=device)
    D = torch.rand(din, generator=gen, device=device) * (1.0 - D_lo) + D_lo
    col = torch.ones(din, device=device)
    if n_out:
        idx = torch.randperm(din, generator=gen, device=device)[:n_out]
        col[idx] = out_scale
    sqD = D.sqrt()
    if token_seed is not None:
        gen.manual_seed(token_seed)
    H = torch.zeros(din, din, dtype=torch.float64, device=device)
    prev = torch.get_float32_matmul_precision()
    torch.set_float32_matmul_precision("highest")
    try:
        done = 0
        while done < tokens:
            m = min(chunk, tokens - done)
            U = torch.randn(m, rank, generator=gen, device=device)
            E = torch.randn(m, din, generator=gen, device=device)
            X = (U @ L.T + E * sqD) * col
            H += (X.T @ X).double()
            done += m
    finally:
        torch.set_float32_matmul_precision(prev)
    H /= tokens
    H += damp * H.diagonal().mean() * torch.eye(din, dtype=torch.float64, device=device)
    return H.float()


def weights_torch(dout, din, w_std, w_out_frac, w_out_mul, law, seed, device):
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    if law == "student_t4":
        # t_4 = N / sqrt(chi2_4 / 4), chi2_4 = sum of four squared normals.
        z = torch.randn(dout, din, generator=gen, device=device)
        chi = torch.zeros(dout, din, device=device)
        for _ in range(4):
            chi += torch.randn(dout, din, generator=gen, device=device) ** 2
        W = z / torch.sqrt(chi / 4.0) * (w_std / math.sqrt(2.0))
    else:
        W = torch.randn(dout, din, generator=gen, device=device) * w_std
    mask = torch.rand(dout, din, generator=gen, device=device) < w_out_frac
    W = torch.where(mask, W * w_out_mul, W)
    return W.float().contiguous()


def config_layer(name, device="cuda", H=None, seed_offset=0):
    """Build one named full-size layer on ``device`` (torch tensors).
    ``seed_offset`` draws another instance of the same shape and statistics
    (0: the named layer itself)."""
    c = CONFIGS[name]
    seed = c["seed"] + 7919 * seed_offset
    if H is None:
        H = hessian_torch(c["din"], c["rank"], c["n_out"], c["out_scale"], c["tokens"],
                          c["D_lo"], seed, device)
    W = weights_torch(c["dout"], c["din"], c["w_std"], c["w_out_frac"], c["w_out_mul"],
                      c["law"], 1000 + seed, device)
    S0, Q0, Z = rtn_host_torch(W, c["bits"], c["g"], c["clip"])
    return Layer(name, W, H, S0, Q0, Z, c["bits"], c["g"], c["K"])


def block_hessians(device="cuda", tokens=262144):
    """The three Hessians of the Llama-2-7B block (attention input, o_proj
    input, down_proj input), built as for the q_proj layer."""
    out = {}
    for key, (din, seed) in BLOCK_HESSIANS.items():
        out[key] = hessian_torch(din, 64, 16 if din == 4096 else 32, 30.0, tokens, 0.05,
                                 seed, device)
    return out


def block_layers(device="cuda", hessians=None, bits=3, g=128, K=10):
    """The seven layers of one Llama-2-7B block with their RTN host state."""
    import torch  # noqa: F401
    hs = hessians if hessians is not None else block_hessians(device)
    layers = []
    for idx, (lname, dout, din, hkey) in enumerate(BLOCK_LLAMA2_7B):
        W = weights_torch(dout, din, 0.015, 0.001, 10.0, "normal", 500 + idx, device)
        S0, Q0, Z = rtn_host_torch(W, bits, g)
        layers.append((hkey, Layer(lname, W, hs[hkey], S0, Q0, Z, bits, g, K)))
    return hs, layers
