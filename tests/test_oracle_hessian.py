"""Pins of the calibration-Hessian oracle against facts the paper and the
mathematics fix, independent of the oracle's own matmul:

* H = A^T A for A = [X; nu I] (Eq. strict_target): the Householder QR of A
  gives R with R^T R = H, a route that never forms a product of columns;
* the H-form objective equals the augmented least-squares objective of
  Eq. adaptive_grid_problem, ||X (what - w)||^2 + nu^2 ||what - w||^2,
  evaluated from the activations themselves;
* a Sylvester-Hadamard activation matrix has the closed form X^T X = n I;
* on integer activations, streaming over token batches is exact and equals
  the brute-force double loop over tokens;
* planted mistakes (a dropped token, a missing cross term, a wrong scale)
  fail at least one of these.
"""
import numpy as np
import pytest

import oracle.jarq_hessian as jh
from oracle import objective, prepare_hessian
from synth import activations_np, integer_activations_np, rtn_host_np


def _sylvester(k):
    Hd = np.array([[1.0]])
    for _ in range(k):
        Hd = np.block([[Hd, Hd], [Hd, -Hd]])
    return Hd


def test_hadamard_closed_form():
    X = _sylvester(4).astype(np.float16)          # 16 tokens x 16 features, entries +-1
    H = jh.accumulate_hessian(X)
    np.testing.assert_array_equal(H, 16.0 * np.eye(16))
    # three of its columns repeated: X^T X has the Gram matrix of the columns
    Xr = X[:, [0, 3, 3, 5]]
    Hr = jh.accumulate_hessian(Xr)
    np.testing.assert_array_equal(Hr, 16.0 * np.array([[1, 0, 0, 0], [0, 1, 1, 0],
                                                        [0, 1, 1, 0], [0, 0, 0, 1]]))


def test_augmented_hessian_is_R_transpose_R_of_householder_qr():
    """Eq. strict_target: the design A = [X; nu I]; its thin QR factor R
    (LAPACK Householder) satisfies R^T R = A^T A = X^T X + nu^2 I."""
    X = activations_np(40, 12, rank=3, n_out=1, seed=3)
    nu = 0.7
    A = np.vstack([X.astype(np.float64), nu * np.eye(12)])
    R = np.linalg.qr(A, mode="r")
    H = jh.augmented_hessian(X, nu)
    np.testing.assert_allclose(R.T @ R, H, rtol=1e-12, atol=1e-12 * np.abs(H).max())


def test_objective_of_accumulated_hessian_is_the_augmented_least_squares_objective():
    """Eq. adaptive_grid_problem, row by row: F_j = ||X (what_j - w_j)||^2 +
    nu^2 ||what_j - w_j||^2 equals r_j^T H r_j with the accumulated H."""
    d, p, g, bits, nu = 32, 6, 8, 3, 0.3
    X = activations_np(200, d, rank=4, n_out=2, seed=4)
    rng = np.random.Generator(np.random.PCG64(5))
    W = (rng.standard_normal((p, d)) * 0.05).astype(np.float32)
    S, Q, Z = rtn_host_np(W, bits, g)
    prep = prepare_hessian(jh.accumulate_hessian(X), g, nu2=nu * nu)
    F = objective(prep, W, S, Q, Z)
    What = np.repeat(S.astype(np.float64), g, axis=1) * (Q.astype(np.float64)
                                                         - np.repeat(Z, g, axis=1))
    Rres = What - W.astype(np.float64)
    direct = (np.sum((X.astype(np.float64) @ Rres.T) ** 2, axis=0)
              + nu * nu * np.sum(Rres ** 2, axis=1))
    np.testing.assert_allclose(F, direct, rtol=1e-10)


def test_streaming_batches_is_exact_and_matches_brute_force():
    X = integer_activations_np(37, 9, amax=8, seed=6)
    one = jh.accumulate_hessian(X)
    H = None
    for a, b in [(0, 5), (5, 6), (6, 30), (30, 37)]:
        H = jh.accumulate_hessian(X[a:b], H)
    np.testing.assert_array_equal(H, one)
    n, d = X.shape
    brute = np.zeros((d, d))
    for i in range(d):
        for j in range(d):
            brute[i, j] = sum(float(X[t, i]) * float(X[t, j]) for t in range(n))
    np.testing.assert_array_equal(one, brute)


def test_scale_and_input_contract():
    X = integer_activations_np(10, 8, seed=7)
    np.testing.assert_array_equal(jh.accumulate_hessian(X, scale=0.25),
                                  0.25 * jh.accumulate_hessian(X))
    with pytest.raises(TypeError):
        jh.accumulate_hessian(X.astype(np.float32))
    with pytest.raises(ValueError):
        jh.accumulate_hessian(X[0])


# ---- planted mistakes ------------------------------------------------------

def _drop_last_token(X, H=None, scale=1.0):
    X64 = np.asarray(X).astype(np.float64)[:-1]
    out = scale * (X64.T @ X64)
    return out if H is None else H + out


def _diagonal_only(X, H=None, scale=1.0):
    X64 = np.asarray(X).astype(np.float64)
    out = scale * np.diag(np.sum(X64 * X64, axis=0))
    return out if H is None else H + out


def _scale_twice(X, H=None, scale=1.0):
    X64 = np.asarray(X).astype(np.float64)
    out = scale * scale * (X64.T @ X64) * 2.0
    return out if H is None else H + out


PINS = [test_hadamard_closed_form,
        test_augmented_hessian_is_R_transpose_R_of_householder_qr,
        test_objective_of_accumulated_hessian_is_the_augmented_least_squares_objective,
        test_streaming_batches_is_exact_and_matches_brute_force]


@pytest.mark.parametrize("mutant", [_drop_last_token, _diagonal_only, _scale_twice])
def test_planted_mistakes_are_caught(monkeypatch, mutant):
    monkeypatch.setattr(jh, "accumulate_hessian", mutant)
    failed = 0
    for pin in PINS:
        try:
            pin()
        except AssertionError:
            failed += 1
    assert failed >= 1, mutant.__name__
