"""Calibration Hessian of a layer (test infrastructure, like jarq_oracle).

TEST INFRASTRUCTURE: only the test-suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this module.

The H-form of the objective uses ``H = A^T A`` for the augmented design
matrix ``A = [X~; nu I]`` of Eq. strict_target, that is
``H = X~^T X~ + nu^2 I`` (App. "Propagation-Corrected Targets and QEP",
where H is written out; ``X~`` stacks the n calibration inputs of the layer,
one token per row, Sec. 3.1).  The paper forms its products from FP16
activations (App. "Metrics"), so the activations enter as float16 values.

* ``accumulate_hessian``: ``H_in + scale * X^T X`` in float64.  Every fp16
  value and every product of two is exact in float64; the library matmul's
  sum over n tokens then carries a relative error of order n 2^-53, far
  below anything the float32 CUDA path can resolve.  ``scale`` lets a caller
  normalise (e.g. 1/n); the paper's H uses 1.
* ``augmented_hessian``: the same plus ``nu^2 I``.
"""
from __future__ import annotations

import numpy as np


def _fp16(X):
    X = np.asarray(X)
    if X.dtype != np.float16:
        raise TypeError("activations are float16 values (App. Metrics)")
    if X.ndim != 2:
        raise ValueError("X is [tokens][features]")
    return X.astype(np.float64)


def accumulate_hessian(X, H=None, scale: float = 1.0):
    """``H + scale * X^T X`` (float64 [d][d]) for float16 X [n][d]."""
    X64 = _fp16(X)
    out = scale * (X64.T @ X64)
    return out if H is None else np.asarray(H, dtype=np.float64) + out


def augmented_hessian(X, nu: float):
    """``A^T A`` for ``A = [X; nu I]`` (Eq. strict_target): ``X^T X + nu^2 I``."""
    H = accumulate_hessian(X)
    return H + (nu * nu) * np.eye(H.shape[0])
