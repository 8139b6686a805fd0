"""Propagation-corrected (mu) target of a layer (test infrastructure, like
jarq_oracle).

TEST INFRASTRUCTURE: only the test-suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this module.

App. "Propagation-Corrected Targets and QEP": keep the design A = [X~; nu I]
of Eq. strict_target and replace the activation part of the target by
Y*(mu) = (1 - mu) X W + mu X~ W (Eq. mu-target; X the full-precision
inputs, X~ the inputs after the quantized preceding layers).  With
H = X~^T X~ + nu^2 I, the unconstrained least-squares solution is

    W_corr = W + (1 - mu) H^{-1} X~^T (X - X~) W          (Eq. w-corr),

and for every What, ||Y(mu) - A What||^2 = ||A (W_corr - What)||^2 + c with
c = ||Y(mu) - A W_corr||^2 (per output row), so refining with the mu-target
is the main problem on W_corr plus the constant c_j.

The inputs are the Gram matrices of the activations (all with the same
normalisation): H (including nu^2 I), K = X~^T X and XX = X^T X, plus nu^2;
so X~^T (X - X~) = K - (H - nu^2 I).  Rows are output channels (W is
[dout][din]).
"""
from __future__ import annotations

import numpy as np

from .jarq_oracle import Options, prepare_hessian, refine_layer


def _f64(*a):
    return [np.asarray(x, dtype=np.float64) for x in a]


def corrected_weights(H, K, W, mu: float, nu2: float):
    """Eq. w-corr, row by row: w_corr = w + (1 - mu) H^{-1} (K - H0) w with
    H0 = H - nu^2 I = X~^T X~; float64, by a dense solve."""
    H, K, W = _f64(H, K, W)
    C = K - (H - nu2 * np.eye(H.shape[0]))
    return W + (1.0 - mu) * np.linalg.solve(H, C @ W.T).T


def target_energy(H, K, XX, W, mu: float, nu2: float):
    """||y_j(mu)||^2 per row for y_j(mu) = [((1 - mu) X + mu X~) w_j; nu w_j]:
    (1-mu)^2 w^T XX w + 2 mu (1-mu) w^T K w + mu^2 w^T H0 w + nu^2 w^T w."""
    H, K, XX, W = _f64(H, K, XX, W)
    H0 = H - nu2 * np.eye(H.shape[0])
    q = lambda M: np.einsum("jd,jd->j", W @ M.T, W)
    return ((1 - mu) ** 2 * q(XX) + 2 * mu * (1 - mu) * q(K) + mu ** 2 * q(H0)
            + nu2 * np.einsum("jd,jd->j", W, W))


def mu_constant(H, K, XX, W, mu: float, nu2: float):
    """c_j = ||y_j(mu) - A w_corr,j||^2 = ||y_j(mu)||^2 - w_corr^T H w_corr
    (Pythagoras: the residual of the least-squares solution is orthogonal
    to the range of A)."""
    Wc = corrected_weights(H, K, W, mu, nu2)
    Hf = np.asarray(H, dtype=np.float64)
    return target_energy(H, K, XX, W, mu, nu2) - np.einsum("jd,jd->j", Wc @ Hf, Wc)


def refine_mu(H, K, XX, W, S0, Q0, Z, bits: int, g: int, mu: float, nu2: float,
              opt: Options = None):
    """JARQ on the mu-target: the main refinement of W_corr with the
    constant c_j carried in the objective.  Returns (Result, W_corr, c)."""
    Wc = corrected_weights(H, K, W, mu, nu2)
    c = mu_constant(H, K, XX, W, mu, nu2)
    prep = prepare_hessian(H, g)
    return refine_layer(prep, Wc, S0, Q0, Z, bits, opt, const=c), Wc, c
