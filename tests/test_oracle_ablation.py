"""Pins of the mechanism-ablation oracle (App. "Refinement Mechanisms").

* The worked example of Prop. multicode-descent (App. G): at the fixed scale
  s0 = 53/52 the host codes (1, 2) are single-code stationary, and the Babai
  proposal from them is (2, 3) with f = 109/270400 < 1/104 = f(q0): the
  multi-code probe accepts it and changes two codes.
* Prop. independent-gap (a): the gap of the independent fit equals
  g^T C^{-1} g with the normalised Gram matrix C and g_i built from the
  other groups' errors; (b): it lies between |g|^2 / lambda_max(C) and
  |g|^2 / lambda_min(C).
* With H block diagonal (groups uncoupled) the independent fit is the joint
  fit, and one coordinate-descent pass reaches it.
* Coordinate descent never raises F and converges to the joint fit.
* The single-code search ends single-code stationary and never raises F.
* Fixed grid keeps the scales and never raises F.
* Planted mistakes fail at least one pin.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle.jarq_ablation as ja
from oracle import objective, prepare_hessian, scale_system
from synth import small_layer

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _frac(x):
    return float(Fraction(x))


def test_multicode_probe_on_the_worked_example():
    ex = json.load(open(os.path.join(GOLDEN, "multicode_example.json")))
    R = np.array([[_frac(v) for v in row] for row in ex["R"]])
    H = R.T @ R
    w = np.array([[_frac(v) for v in ex["w"]]])
    s0 = _frac(ex["s0"])
    q0 = np.array([ex["q0"]], dtype=np.uint8)
    Z = np.array([[ex["z"]]], dtype=np.int32)
    prep = prepare_hessian(H, 2)
    out = ja.multicode_probe(prep, w, np.array([[s0]]), q0, Z, ex["bits"], 0)
    assert out["moves"][0] == 0                       # already single-code stationary
    np.testing.assert_array_equal(out["q_search"][0], ex["q0"])
    assert out["accepted"][0] and out["changed"][0] == 2
    f_plus = objective(prep, w, np.array([[s0]]), np.array([ex["q_plus"]]), Z)[0]
    assert abs(f_plus - _frac(ex["f_s0_qplus"])) <= 1e-15
    assert abs(out["dF"][0] - (_frac(ex["f_s0_qplus"]) - _frac(ex["phi_q0"]))) <= 1e-15


def _layer(seed=3, din=96, dout=10, g=16):
    return small_layer(din, dout, g, 3, seed=seed)


def test_independent_gap_matches_the_proposition():
    lay = _layer()
    prep = prepare_hessian(lay.H, lay.g)
    g, G, H = lay.g, lay.din // lay.g, prep.H
    Si = ja.independent_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    Sj = ja.joint_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    f_ind = objective(prep, lay.W, Si, lay.Q0, lay.Z)
    f_min = objective(prep, lay.W, Sj, lay.Q0, lay.Z)
    Gram, _ = scale_system(prep, lay.W, lay.Q0, lay.Z)
    C = lay.Q0.astype(np.float64) - np.repeat(lay.Z, g, axis=1)
    E = lay.W.astype(np.float64) - np.repeat(Si, g, axis=1) * C        # e_h = w_h - s~_h c_h
    for j in range(lay.dout):
        d = np.sqrt(np.diag(Gram[j]))
        Cn = Gram[j] / np.outer(d, d)
        ghat = np.zeros(G)
        for i in range(G):
            si = slice(i * g, (i + 1) * g)
            for h in range(G):
                if h == i:
                    continue
                sh = slice(h * g, (h + 1) * g)
                ghat[i] += C[j, si] @ H[si, sh] @ E[j, sh] / d[i]
        delta = ghat @ np.linalg.solve(Cn, ghat)
        gap = f_ind[j] - f_min[j]
        assert abs(gap - delta) <= 1e-9 * f_min[j] + 1e-12, (j, gap, delta)
        lam = np.linalg.eigvalsh(Cn)
        gg = ghat @ ghat
        assert gg / lam[-1] * (1 - 1e-9) <= gap <= gg / lam[0] * (1 + 1e-9)


def test_uncoupled_groups_make_the_fits_agree():
    lay = _layer(seed=4)
    g = lay.g
    Hb = np.zeros_like(lay.H, dtype=np.float64)
    for i in range(lay.din // g):
        si = slice(i * g, (i + 1) * g)
        Hb[si, si] = lay.H[si, si]
    prep = prepare_hessian(Hb, g)
    Sj = ja.joint_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    Si = ja.independent_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    Sc = ja.coordinate_descent_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z, passes=1)
    np.testing.assert_allclose(Si, Sj, rtol=1e-10)
    np.testing.assert_allclose(Sc, Sj, rtol=1e-10)


def test_coordinate_descent_descends_and_converges():
    lay = _layer(seed=5)
    prep = prepare_hessian(lay.H, lay.g)
    F = [objective(prep, lay.W, lay.S0, lay.Q0, lay.Z)]
    for p in range(1, 6):
        S = ja.coordinate_descent_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z, passes=p)
        F.append(objective(prep, lay.W, S, lay.Q0, lay.Z))
    F = np.array(F)
    assert np.all(F[1:] <= F[:-1] * (1 + 1e-12))
    Sj = ja.joint_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    S400 = ja.coordinate_descent_scales(prep, lay.W, lay.S0, lay.Q0, lay.Z, passes=400)
    f_j = objective(prep, lay.W, Sj, lay.Q0, lay.Z)
    f_c = objective(prep, lay.W, S400, lay.Q0, lay.Z)
    assert np.all(f_c - f_j <= 1e-8 * f_j)
    gaps = ja.scale_fit_gaps(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    assert np.all(gaps["gap_independent"] >= -1e-6) and np.all(gaps["gap_coordinate"] >= -1e-6)


def test_single_code_search_is_stationary_and_descends():
    lay = _layer(seed=6, din=64, dout=6, g=16)
    prep = prepare_hessian(lay.H, lay.g)
    g, qmax = lay.g, (1 << lay.bits) - 1
    H = prep.H
    for i in range(lay.din // g):
        out = ja.multicode_probe(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits, i)
        si = slice(i * g, (i + 1) * g)
        Qs = lay.Q0.astype(np.float64).copy()
        Qs[:, si] = out["q_search"]
        F0 = objective(prep, lay.W, lay.S0, lay.Q0, lay.Z)
        F1 = objective(prep, lay.W, lay.S0, Qs, lay.Z)
        assert np.all(F1 <= F0 * (1 + 1e-12))
        C = Qs - np.repeat(lay.Z, g, axis=1)
        Rr = lay.W - np.repeat(lay.S0.astype(np.float64), g, axis=1) * C
        for j in range(lay.dout):
            hr = Rr[j] @ H[:, si]
            assert ja.is_single_code_stationary(H[si, si], hr, float(lay.S0[j, i]), Qs[j, si], qmax)


def test_fixed_grid_keeps_the_scales_and_descends():
    lay = _layer(seed=7)
    prep = prepare_hessian(lay.H, lay.g)
    Q, hist = ja.refine_fixed_grid(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits, 3)
    F0 = objective(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    h = np.array([F0] + hist)
    assert np.all(h[1:] <= h[:-1] * (1 + 1e-12))
    np.testing.assert_allclose(hist[-1], objective(prep, lay.W, lay.S0, Q, lay.Z))


# ---- planted mistakes ------------------------------------------------------

def _indep_full_target(prep, W, S0, Q, Z):
    # the estimator the paper explicitly sets aside: each scale fitted alone
    # to the full target, b_i^T y / ||b_i||^2
    g, G, H = prep.g, prep.G, prep.H
    W = np.asarray(W, dtype=np.float64)
    C = ja._codes(Q, Z, g)
    S = np.array(S0, dtype=np.float64, copy=True)
    HW = W @ H
    for i in range(G):
        si = slice(i * g, (i + 1) * g)
        S[:, i] = (np.einsum("jk,jk->j", C[:, si], HW[:, si])
                   / np.einsum("jk,jk->j", C[:, si] @ H[si, si], C[:, si]))
    return S


def _cd_stale_gradient(prep, W, S0, Q, Z, passes=3):
    Gram, rhs = scale_system(prep, W, Q, Z)
    S = np.array(S0, dtype=np.float64, copy=True)
    for j in range(S.shape[0]):
        grad = rhs[j] - Gram[j] @ S[j]
        for _ in range(passes):
            for i in range(S.shape[1]):
                S[j, i] += grad[i] / Gram[j, i, i]
    return S


def _search_without_update(Hii, hr, s, q, z, qmax):
    q = np.array(q, dtype=np.float64, copy=True)
    cand = np.arange(qmax + 1, dtype=np.float64)
    for l in range(q.size):
        delta = s * (cand - q[l])
        dF = -2.0 * delta * hr[l] + delta * delta * Hii[l, l]
        k = int(np.argmin(dF))
        if dF[k] < 0.0:
            q[l] = cand[k]
    return q, hr, 0


PINS = [test_multicode_probe_on_the_worked_example, test_independent_gap_matches_the_proposition,
        test_uncoupled_groups_make_the_fits_agree, test_coordinate_descent_descends_and_converges,
        test_single_code_search_is_stationary_and_descends]


@pytest.mark.parametrize("name,patch", [
    ("independent_full_target", ("independent_scales", _indep_full_target)),
    ("cd_stale_gradient", ("coordinate_descent_scales", _cd_stale_gradient)),
    ("search_no_update", ("single_code_search", _search_without_update)),
])
def test_planted_mistakes_are_caught(monkeypatch, name, patch):
    monkeypatch.setattr(ja, patch[0], patch[1])
    failed = 0
    for pin in PINS:
        try:
            pin()
        except (AssertionError, np.linalg.LinAlgError):
            failed += 1
    assert failed >= 1, name
