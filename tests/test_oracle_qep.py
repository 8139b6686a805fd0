"""Pins of the mu-target oracle (App. "Propagation-Corrected Targets and
QEP") against routes that never use its formula:

* W_corr is the least-squares solution of min ||Y(mu) - A What|| over real
  matrices, with A = [X~; nu I] and Y(mu) = [((1-mu) X + mu X~) W; nu W]
  built explicitly from the activations (LAPACK lstsq) -- Eq. w-corr;
* the residual Y(mu) - A W_corr is orthogonal to the range of A;
* the objective the oracle refines (main objective on W_corr plus c_j)
  equals ||y_j(mu) - A what_j||^2 evaluated from the activations;
* mu = 1 gives back the main target (W_corr = W, c = 0);
* the refinement on the mu-target descends at every recorded objective;
* planted mistakes fail at least one pin.
"""
import numpy as np
import pytest

import oracle.jarq_qep as jq
from oracle import Options, objective, prepare_hessian
from synth.qep import drifted_activations_np, mu_layer
from synth import rtn_host_np

D, P, G_SIZE, N_TOK = 24, 5, 8, 120


def _case(seed=3, drift=0.08):
    Xq, Xf = drifted_activations_np(N_TOK, D, drift=drift, rank=3, seed=seed)
    A_ = Xq.astype(np.float64)
    B_ = Xf.astype(np.float64)
    nu2 = 0.05 * np.mean(np.sum(A_ * A_, axis=0))
    H = A_.T @ A_ + nu2 * np.eye(D)
    K = A_.T @ B_
    XX = B_.T @ B_
    rng = np.random.Generator(np.random.PCG64(seed))
    W = rng.standard_normal((P, D)) * 0.05
    return A_, B_, H, K, XX, W, nu2


def _design(A_, B_, W, mu, nu2):
    """Explicit A = [X~; nu I] and Y(mu) (Eqs. strict_target, mu-target), paper layout."""
    nu = np.sqrt(nu2)
    A = np.vstack([A_, nu * np.eye(A_.shape[1])])
    Y = np.vstack([((1 - mu) * B_ + mu * A_) @ W.T, nu * W.T])
    return A, Y


@pytest.mark.parametrize("mu", [0.0, 0.5, 0.9])
def test_w_corr_is_the_least_squares_solution(mu):
    A_, B_, H, K, XX, W, nu2 = _case()
    A, Y = _design(A_, B_, W, mu, nu2)
    ls = np.linalg.lstsq(A, Y, rcond=None)[0].T
    Wc = jq.corrected_weights(H, K, W, mu, nu2)
    np.testing.assert_allclose(Wc, ls, rtol=1e-9, atol=1e-12)
    # the residual is orthogonal to the range of A
    R = Y - A @ Wc.T
    assert np.abs(A.T @ R).max() <= 1e-9 * np.abs(A.T @ Y).max()


@pytest.mark.parametrize("mu", [0.0, 0.5])
def test_mu_objective_is_the_augmented_objective(mu):
    A_, B_, H, K, XX, W, nu2 = _case(seed=4)
    A, Y = _design(A_, B_, W, mu, nu2)
    S, Q, Z = rtn_host_np(W.astype(np.float32), 3, G_SIZE)
    What = np.repeat(S.astype(np.float64), G_SIZE, axis=1) * (
        Q.astype(np.float64) - np.repeat(Z, G_SIZE, axis=1))
    direct = np.sum((Y - A @ What.T) ** 2, axis=0)
    Wc = jq.corrected_weights(H, K, W, mu, nu2)
    c = jq.mu_constant(H, K, XX, W, mu, nu2)
    F = objective(prepare_hessian(H, G_SIZE), Wc, S, Q, Z) + c
    np.testing.assert_allclose(F, direct, rtol=1e-9)
    # ||y||^2 from the Gram matrices equals the explicit one
    np.testing.assert_allclose(jq.target_energy(H, K, XX, W, mu, nu2),
                               np.sum(Y ** 2, axis=0), rtol=1e-10)


def test_mu_one_is_the_main_target():
    A_, B_, H, K, XX, W, nu2 = _case(seed=5)
    np.testing.assert_array_equal(jq.corrected_weights(H, K, W, 1.0, nu2), W)
    c = jq.mu_constant(H, K, XX, W, 1.0, nu2)
    assert np.all(np.abs(c) <= 1e-10 * jq.target_energy(H, K, XX, W, 1.0, nu2))


def test_refine_mu_descends_and_reports_the_mu_objective():
    lay = mu_layer(64, 12, 16, 3, tokens=600, drift=0.1, seed=8)
    res, Wc, c = jq.refine_mu(lay.H, lay.K, lay.XX, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits,
                              lay.g, 0.5, lay.nu2, Options(max_iters=4, early_stop=False))
    hist = np.array(res.L_hist)
    assert np.all(hist[1:] <= hist[:-1] * (1 + 1e-12))
    assert np.all(res.L_final <= res.L_host * (1 + 1e-12))
    # L_final is the mu-objective of the returned state, computed from the activations
    A_, B_ = lay.Xq.astype(np.float64), lay.Xf.astype(np.float64)
    n = A_.shape[0]
    A, Y = _design(A_ / np.sqrt(n), B_ / np.sqrt(n), lay.W.astype(np.float64), 0.5, lay.nu2)
    What = np.repeat(res.S, lay.g, axis=1) * (res.Q - np.repeat(lay.Z, lay.g, axis=1))
    direct = np.sum((Y - A @ What.T) ** 2, axis=0)
    # H, K, XX were rounded to float32 once: agreement to that precision
    np.testing.assert_allclose(res.L_final, direct, rtol=2e-5)


# ---- planted mistakes ------------------------------------------------------

def _sign_flipped(H, K, W, mu, nu2):
    H, K, W = [np.asarray(x, dtype=np.float64) for x in (H, K, W)]
    C = K - (H - nu2 * np.eye(H.shape[0]))
    return W - (1.0 - mu) * np.linalg.solve(H, C @ W.T).T


def _mu_for_one_minus_mu(H, K, W, mu, nu2):
    H, K, W = [np.asarray(x, dtype=np.float64) for x in (H, K, W)]
    C = K - (H - nu2 * np.eye(H.shape[0]))
    return W + mu * np.linalg.solve(H, C @ W.T).T


def _ridge_counted_in_cross_term(H, K, W, mu, nu2):
    H, K, W = [np.asarray(x, dtype=np.float64) for x in (H, K, W)]
    return W + (1.0 - mu) * np.linalg.solve(H, (K - H) @ W.T).T


PINS = [lambda: test_w_corr_is_the_least_squares_solution(0.0),
        lambda: test_w_corr_is_the_least_squares_solution(0.5),
        lambda: test_mu_objective_is_the_augmented_objective(0.5),
        test_mu_one_is_the_main_target]


@pytest.mark.parametrize("name,patch", [
    ("sign", ("corrected_weights", _sign_flipped)),
    ("mu", ("corrected_weights", _mu_for_one_minus_mu)),
    ("ridge", ("corrected_weights", _ridge_counted_in_cross_term)),
    ("no_constant", ("mu_constant", lambda H, K, XX, W, mu, nu2: np.zeros(W.shape[0]))),
])
def test_planted_mistakes_are_caught(monkeypatch, name, patch):
    monkeypatch.setattr(jq, patch[0], patch[1])
    failed = 0
    for pin in PINS:
        try:
            pin()
        except AssertionError:
            failed += 1
    assert failed >= 1, name
