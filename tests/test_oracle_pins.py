"""Pins of the float64 oracle against what the paper and mathematics fix.

Each test pins one part of the oracle to something other than itself: the
paper's worked examples with exact rationals (App. G), brute force on tiny
groups, closed forms (G = 1, stationarity), the paper's theorems as
invariants (Thm. descent, Cor. host, Props. babai-vs-rounding and
stable-quality), and an independent paper-literal QR-form implementation.
"""
import itertools
import json
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import (FP32_EPS, Options, babai_proposal, canonicalize, code_sweep, dequantize,
                    group_target, objective, prepare_hessian, refine_layer, scale_system,
                    solve_scales)
from oracle.jarq_qr_literal import refine_columns
from synth import small_layer, tiny_layer


def F(x):
    return float(Fraction(x))


def load(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as fh:
        return json.load(fh)


# ---------------------------------------------------------------------------
# Worked example of Prop. multicode-descent (App. G)
# ---------------------------------------------------------------------------

def multicode_setup(ex):
    R = np.array([[F(x) for x in row] for row in ex["R"]])
    H = R.T @ R
    W = np.array([[F(x) for x in ex["w"]]])
    return R, H, W


def test_multicode_single_code_neighbours(golden_dir):
    """phi(q) = min_s F(s, q) for q0 and all six single-code neighbours
    (Table single-code-example) equals the oracle's scale solve + objective."""
    ex = load(golden_dir, "multicode_example.json")
    _, H, W = multicode_setup(ex)
    prep = prepare_hessian(H, 2)
    Z = np.zeros((1, 1), dtype=np.int32)
    cases = [{"q": ex["q0"], "phi": ex["phi_q0"]}] + ex["single_code_neighbours"]
    for case in cases:
        Q = np.array([case["q"]])
        Gram, rhs = scale_system(prep, W, Q, Z)
        s, ridge, ok = solve_scales(Gram[0], rhs[0], Options())
        assert ok and not ridge
        phi = objective(prep, W, s[None, :], Q, Z)[0]
        assert phi == pytest.approx(F(case["phi"]), rel=1e-12, abs=1e-15), case
    # the host state's scale
    Gram, rhs = scale_system(prep, W, np.array([ex["q0"]]), Z)
    s, _, _ = solve_scales(Gram[0], rhs[0], Options())
    assert s[0] == pytest.approx(F(ex["s0"]), rel=1e-14)


def test_multicode_babai_step_and_refit(golden_dir):
    """Babai at s0 gives pre-round values 156/53, 107/53 -> q+ = (2,3),
    f(s0, q+) = 109/270400; the next refit gives s = 1 and F = 0."""
    ex = load(golden_dir, "multicode_example.json")
    _, H, W = multicode_setup(ex)
    prep = prepare_hessian(H, 2)
    Z = np.zeros((1, 1), dtype=np.int32)
    Q0 = np.array([ex["q0"]], dtype=np.uint8)
    S0 = np.array([[F(ex["s0"])]])
    trace = []
    # the worked example is exact arithmetic: keep float64 scales
    res = refine_layer(prep, W, S0, Q0, Z, ex["bits"],
                       Options(max_iters=2, early_stop=False, fp32_scales=False), trace=trace)
    scale1, babai1, sweep1, scale2 = trace[0], trace[1], trace[2], trace[3]
    assert scale1["S"][0, 0] == pytest.approx(F(ex["s0"]), rel=1e-14)
    assert scale1["L"][0] == pytest.approx(F(ex["phi_q0"]), rel=1e-12)
    zx = babai1["z"][0] + babai1["x"][0]
    assert zx[1] == pytest.approx(F(ex["babai_preround_at_s0"]["2"]), rel=1e-13)
    assert zx[0] == pytest.approx(F(ex["babai_preround_at_s0"]["1"]), rel=1e-13)
    assert list(babai1["proposal"][0]) == ex["q_plus"]
    assert babai1["accepted"][0]
    assert sweep1["F"][0] == pytest.approx(F(ex["f_s0_qplus"]), rel=1e-11)
    assert scale2["S"][0, 0] == pytest.approx(F(ex["s_plus"]), rel=1e-13)
    assert abs(scale2["L"][0]) < 1e-20
    assert list(res.Q[0]) == ex["q_plus"]
    assert abs(res.L_final[0]) < 1e-20


# ---------------------------------------------------------------------------
# Worked example of Prop. grid-staleness (App. G)
# ---------------------------------------------------------------------------

def staleness_setup(ex):
    rho = F(ex["rho"])
    H = np.array([[1.0, rho], [rho, 1.0]])
    W = np.array([[F(x) for x in ex["w"]]])
    return H, W


def test_staleness_host_grid_optimum(golden_dir):
    """At (s0, q0): F0 = 16889/50000, q0 minimises F(s0, .) over all 16 codes
    and the runner-up is (0,2) with 19241/50000; Babai at s0 returns q0."""
    ex = load(golden_dir, "grid_staleness_example.json")
    H, W = staleness_setup(ex)
    prep = prepare_hessian(H, 2)
    Z = np.zeros((1, 1), dtype=np.int32)
    s0 = np.array([[F(ex["s0"])]])
    vals = {}
    for q in itertools.product(range(4), repeat=2):
        vals[q] = objective(prep, W, s0, np.array([q]), Z)[0]
    order = sorted(vals, key=vals.get)
    assert order[0] == tuple(ex["q0"])
    assert vals[order[0]] == pytest.approx(F(ex["F0"]), rel=1e-13)
    assert order[1] == tuple(ex["second_best_at_s0"]["q"])
    assert vals[order[1]] == pytest.approx(F(ex["second_best_at_s0"]["F"]), rel=1e-13)
    # codes-only sweep on the host grid: the proposal is q0 itself
    Q = np.array([ex["q0"]], dtype=np.int64)
    trace = []
    dF, nacc = code_sweep(prep, W, s0, Q, Z, ex["bits"], Options(), trace=trace)
    zx = trace[0]["z"][0] + trace[0]["x"][0]
    assert zx[1] == pytest.approx(F(ex["babai_preround_at_s0"]["2"]), rel=1e-13)
    assert zx[0] == pytest.approx(F(ex["babai_preround_at_s0"]["1"]), rel=1e-13)
    assert list(trace[0]["proposal"][0]) == ex["q0"]
    assert nacc[0] == 0 and list(Q[0]) == ex["q0"]


def test_staleness_refit_unlocks_descent(golden_dir):
    """Refit -> s1 = 197/200; Babai (pre-round 310/197, 588/4925) -> (0,2)
    with F = 3087/31250; refit -> s2 = 4631/5000, F = 132741/1562500; the
    proposal at s2 repeats (0,2) and is not accepted."""
    ex = load(golden_dir, "grid_staleness_example.json")
    H, W = staleness_setup(ex)
    prep = prepare_hessian(H, 2)
    Z = np.zeros((1, 1), dtype=np.int32)
    trace = []
    res = refine_layer(prep, W, np.array([[F(ex["s0"])]]), np.array([ex["q0"]], dtype=np.uint8), Z,
                       ex["bits"], Options(max_iters=2, early_stop=False, fp32_scales=False),
                       trace=trace)
    sc1, b1, sw1, sc2, b2, sw2 = trace
    assert res.L_host[0] == pytest.approx(F(ex["F0"]), rel=1e-13)
    assert sc1["S"][0, 0] == pytest.approx(F(ex["s1"]), rel=1e-14)
    assert sc1["L"][0] == pytest.approx(F(ex["F_s1_q0"]), rel=1e-13)
    zx = b1["z"][0] + b1["x"][0]
    assert zx[1] == pytest.approx(F(ex["babai_preround_at_s1"]["2"]), rel=1e-13)
    assert zx[0] == pytest.approx(F(ex["babai_preround_at_s1"]["1"]), rel=1e-12)
    assert list(b1["proposal"][0]) == ex["q_plus"] and b1["accepted"][0]
    assert sw1["F"][0] == pytest.approx(F(ex["F_s1_qplus"]), rel=1e-13)
    assert sc2["S"][0, 0] == pytest.approx(F(ex["s2"]), rel=1e-14)
    assert sc2["L"][0] == pytest.approx(F(ex["F_s2_qplus"]), rel=1e-13)
    assert list(b2["proposal"][0]) == ex["q_plus"]
    assert not b2["accepted"][0] and b2["dF"][0] == 0.0
    assert list(res.Q[0]) == ex["q_plus"]
    assert res.L_final[0] == pytest.approx(F(ex["F_s2_qplus"]), rel=1e-13)


def test_scales_are_stored_as_correctly_rounded_float32(golden_dir):
    """App. E: the scale system is solved in single precision.  With the
    default options every stored scale is the float32 value nearest to the
    exact solve: on the staleness example s1 = 197/200 and s2 = 4631/5000
    are stored as float32(197/200) and float32(4631/5000), and the objective
    L^(k) is evaluated at those float32 scales."""
    ex = load(golden_dir, "grid_staleness_example.json")
    H, W = staleness_setup(ex)
    prep = prepare_hessian(H, 2)
    Z = np.zeros((1, 1), dtype=np.int32)
    trace = []
    refine_layer(prep, W, np.array([[F(ex["s0"])]]), np.array([ex["q0"]], dtype=np.uint8), Z,
                 ex["bits"], Options(max_iters=2, early_stop=False), trace=trace)
    sc1, _, _, sc2, _, _ = trace
    s1 = float(np.float32(F(ex["s1"])))
    s2 = float(np.float32(F(ex["s2"])))
    assert s1 != F(ex["s1"]) and s2 != F(ex["s2"])   # neither is a float32
    assert sc1["S"][0, 0] == s1
    assert sc2["S"][0, 0] == s2
    assert sc1["L"][0] == pytest.approx(objective(prep, W, np.array([[s1]]),
                                                  np.array([ex["q0"]]), Z)[0], rel=1e-15)
    # the float32 rounding moves the objective by a second-order amount only
    assert sc1["L"][0] == pytest.approx(F(ex["F_s1_q0"]), rel=1e-12)


# ---------------------------------------------------------------------------
# Babai recursion: brute force, nearest-plane bound, expectation
# ---------------------------------------------------------------------------

def group_error(Hii, t, s, z, q):
    """E(q) - const = s^2 c^T H_ii c - 2 s c^T t, c = q - z (Eq. group_bils)."""
    c = np.asarray(q, dtype=np.float64) - z
    return s * s * c @ Hii @ c - 2.0 * s * c @ t


def test_babai_equals_brute_force_when_block_diagonal():
    """With diagonal H_ii the bounded Babai proposal is the exact minimiser of
    Eq. group_bils over all 4^4 codes (group size 4, 2-bit)."""
    rng = np.random.default_rng(11)
    codes = np.array(list(itertools.product(range(4), repeat=4)), dtype=np.float64)
    for _ in range(300):
        Hii = np.diag(rng.uniform(0.2, 3.0, 4))
        R = np.sqrt(Hii)
        s = rng.uniform(0.2, 1.5) * rng.choice([-1, 1])
        z = int(rng.integers(0, 4))
        t = rng.normal(0, 2.0, 4)
        v = np.linalg.solve(R.T, t) / s
        q, _ = babai_proposal(R, v[None, :], np.array([float(z)]), 3)
        errs = np.array([group_error(Hii, t, s, z, c) for c in codes])
        best = errs.min()
        assert group_error(Hii, t, s, z, q[0]) == pytest.approx(best, abs=1e-12)


def test_babai_never_beats_brute_force_and_bound():
    """General H_ii: brute force lower-bounds Babai; without clipping every
    entry of v - R(q - z) is at most |R_ll|/2 (Prop. babai-vs-rounding (a))."""
    rng = np.random.default_rng(12)
    codes = np.array(list(itertools.product(range(4), repeat=4)), dtype=np.float64)
    n_unclipped = 0
    for _ in range(300):
        M = rng.normal(size=(8, 4))
        Hii = M.T @ M + 0.1 * np.eye(4)
        R = np.linalg.cholesky(Hii).T
        s = rng.uniform(0.3, 1.0)
        z = int(rng.integers(0, 4))
        t = rng.normal(0, 1.0, 4)
        v = np.linalg.solve(R.T, t) / s
        q, x = babai_proposal(R, v[None, :], np.array([float(z)]), 3)
        eb = group_error(Hii, t, s, z, q[0])
        best = min(group_error(Hii, t, s, z, c) for c in codes)
        assert best <= eb + 1e-12
        unclipped = np.all((z + x[0] >= -0.5) & (z + x[0] <= 3.5))
        if unclipped:
            n_unclipped += 1
            res = v - R @ (q[0] - z)
            assert np.all(np.abs(res) <= np.abs(np.diag(R)) / 2 + 1e-12)
    assert n_unclipped > 30


def test_babai_expected_gain_over_rounding():
    """Prop. babai-vs-rounding (b): with no code bounds and uniform fractional
    parts, E|v - R c|^2 is sum R_ll^2 / 12 for Babai and ||R||_F^2 / 12 for
    coordinatewise rounding of the real minimiser."""
    rng = np.random.default_rng(13)
    g = 6
    M = rng.normal(size=(12, g))
    R = np.linalg.cholesky(M.T @ M + 0.5 * np.eye(g)).T
    n = 60000
    xi = rng.uniform(40, 80, (n, g))       # real minimisers, z = 0, far from the bounds
    v = xi @ R.T                            # v = R xi
    q, _ = babai_proposal(R, v, np.zeros(n), 10 ** 9)
    qb = q - 0.0
    eb = np.mean(np.sum((v - qb @ R.T) ** 2, axis=1))
    er = np.mean(np.sum((v - np.rint(xi) @ R.T) ** 2, axis=1))
    assert eb == pytest.approx(np.sum(np.diag(R) ** 2) / 12, rel=0.03)
    assert er == pytest.approx(np.sum(R ** 2) / 12, rel=0.03)
    assert er - eb == pytest.approx(np.sum(np.triu(R, 1) ** 2) / 12, rel=0.1)


def test_babai_row_sign_invariance():
    """QR factors differ from the Cholesky factor by row signs; flipping the
    signs of rows of R and of v leaves the proposal unchanged."""
    rng = np.random.default_rng(14)
    M = rng.normal(size=(16, 8))
    R = np.linalg.cholesky(M.T @ M).T
    v = rng.normal(0, 3, (50, 8))
    z = rng.integers(0, 8, 50).astype(np.float64)
    q1, _ = babai_proposal(R, v, z, 7)
    D = np.diag(rng.choice([-1.0, 1.0], 8))
    q2, _ = babai_proposal(D @ R, v @ D, z, 7)
    assert np.array_equal(q1, q2)


# ---------------------------------------------------------------------------
# Scale solve: closed forms
# ---------------------------------------------------------------------------

def test_single_group_scale_is_scalar_least_squares():
    """G = 1: the joint fit reduces to s = c^T H w / c^T H c."""
    lay = small_layer(16, 10, 16, 3, seed=3, rank=4, tokens=200)
    prep = prepare_hessian(lay.H, 16)
    Gram, rhs = scale_system(prep, lay.W, lay.Q0, lay.Z)
    H = prep.H
    for j in range(10):
        c = lay.Q0[j].astype(np.float64) - lay.Z[j, 0]
        w = lay.W[j].astype(np.float64)
        s, _, ok = solve_scales(Gram[j], rhs[j], Options())
        assert ok
        assert s[0] == pytest.approx((c @ H @ w) / (c @ H @ c), rel=1e-12)


def test_scale_solve_is_stationary():
    """Prop. joint-scale-gap: the normal equations make the gradient in the
    scales vanish, c_i^T (H r)_i = 0 for every group, and any other scales
    are worse by exactly ||B (s~ - s*)||^2."""
    lay = small_layer(256, 32, 32, 3, seed=4)
    prep = prepare_hessian(lay.H, lay.g)
    Gram, rhs = scale_system(prep, lay.W, lay.Q0, lay.Z)
    S = np.zeros_like(lay.S0, dtype=np.float64)
    for j in range(lay.dout):
        s, _, ok = solve_scales(Gram[j], rhs[j], Options())
        assert ok
        S[j] = s
    C = lay.Q0.astype(np.float64) - np.repeat(lay.Z, lay.g, 1)
    r = lay.W.astype(np.float64) - np.repeat(S, lay.g, 1) * C
    Hr = r @ prep.H
    grad = (C * Hr).reshape(lay.dout, lay.G, lay.g).sum(-1)
    scale = np.abs(C * (lay.W.astype(np.float64) @ prep.H)).reshape(lay.dout, lay.G, lay.g).sum(-1)
    assert np.max(np.abs(grad) / scale) < 1e-10
    F_opt = objective(prep, lay.W, S, lay.Q0, lay.Z)
    F_host = objective(prep, lay.W, lay.S0, lay.Q0, lay.Z)
    ds = lay.S0.astype(np.float64) - S
    gap = np.einsum("ji,jih,jh->j", ds, Gram, ds)
    np.testing.assert_allclose(F_host - F_opt, gap, rtol=1e-8, atol=1e-14)


def test_ridge_branch_on_zero_group():
    """App. E 'Solving for scales': a group whose codes all equal its zero
    point gives a singular Gram matrix; the ridge is added and the solve
    still returns finite scales (that group's scale is 0)."""
    lay = small_layer(64, 4, 16, 3, seed=5, rank=4, tokens=400)
    Q = lay.Q0.copy()
    Q[1, 16:32] = lay.Z[1, 1]
    prep = prepare_hessian(lay.H, lay.g)
    res = refine_layer(prep, lay.W, lay.S0, Q, lay.Z, 3, Options(max_iters=1, early_stop=False))
    assert res.ridge_hits[1] >= 1
    assert np.all(np.isfinite(res.S))
    assert res.ridge_hits[0] == 0 and res.ridge_hits[2] == 0


# ---------------------------------------------------------------------------
# Whole-loop invariants (Thm. descent, Cor. host, Prop. stable-quality)
# ---------------------------------------------------------------------------

def test_monotone_descent_every_half_step():
    """Thm. descent (i): F never increases at a scale update or a code update
    (no ridge triggered on this layer)."""
    lay = tiny_layer()
    prep = prepare_hessian(lay.H, lay.g)
    trace = []
    res = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits,
                       Options(max_iters=6, early_stop=False), trace=trace)
    assert res.ridge_hits.sum() == 0
    prev = res.L_host.copy()
    for ev in trace:
        if ev["kind"] == "scale":
            cur = ev["L"]
        elif ev["kind"] == "sweep":
            cur = ev["F"]
        else:
            continue
        assert np.all(cur <= prev[ev["rows"]] * (1 + 1e-12) + 1e-15)
        prev = prev.copy()
        prev[ev["rows"]] = cur
    # Cor. host
    assert np.all(res.L_final <= res.L_host * (1 + 1e-12))
    assert res.L_final.sum() < 0.5 * res.L_host.sum()


def test_accepted_proposals_strictly_decrease():
    """Sec. 3.3.2: a proposal is kept only if it strictly lowers the group
    objective; the sum of accepted dF equals the sweep's change of F."""
    lay = small_layer(256, 24, 64, 3, seed=6)
    prep = prepare_hessian(lay.H, lay.g)
    S = lay.S0.astype(np.float64)
    Q = lay.Q0.astype(np.int64)
    F0 = objective(prep, lay.W, S, Q, lay.Z)
    trace = []
    dF, nacc = code_sweep(prep, lay.W, S, Q, lay.Z, lay.bits, Options(), trace=trace)
    F1 = objective(prep, lay.W, S, Q, lay.Z)
    np.testing.assert_allclose(F1 - F0, dF, rtol=1e-9, atol=1e-12)
    for ev in trace:
        assert np.all(ev["dF"][ev["accepted"]] < 0)
    assert nacc.sum() > 0


def test_fixed_point_and_early_stop():
    """Thm. descent (iii) and App. G 'Early stopping': with a large budget and
    no early stop the codes stop changing; with early stop a row stops at most
    one iteration after its codes last changed."""
    lay = small_layer(128, 16, 32, 3, seed=8)
    prep = prepare_hessian(lay.H, lay.g)
    res = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits,
                       Options(max_iters=40, early_stop=False))
    res2 = refine_layer(prep, lay.W, res.S, res.Q, lay.Z, lay.bits,
                        Options(max_iters=2, early_stop=False))
    assert np.array_equal(res.Q, res2.Q)
    np.testing.assert_allclose(res2.S, res.S, rtol=1e-9)
    # with tau = 0 a row stops exactly when L^{(k)} equals L^{(k-1)}, which
    # happens one iteration after its codes stop changing; its codes then
    # equal those of the long run without early stopping
    res3 = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits,
                        Options(max_iters=40, early_stop=True, tau=0.0))
    assert np.all(res3.iters < 40)
    assert np.array_equal(res3.Q, res.Q)
    # the early-stopped state is itself a fixed point
    res4 = refine_layer(prep, lay.W, res3.S, res3.Q, lay.Z, lay.bits,
                        Options(max_iters=1, early_stop=False))
    assert np.array_equal(res4.Q, res3.Q)


def test_stable_point_quality_bound():
    """Prop. stable-quality: at a scale-optimal, Babai-stable point, a group
    whose proposal needs no clipping has conditional error within
    s^2 sum R_ll^2 / 4 of its best real-valued fit."""
    lay = small_layer(128, 16, 32, 4, seed=9)
    prep = prepare_hessian(lay.H, lay.g)
    res = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits,
                       Options(max_iters=60, early_stop=False))
    # verify stability: one more sweep at the same scales accepts nothing
    Q = res.Q.copy()
    trace = []
    _, nacc = code_sweep(prep, lay.W, res.S, Q, lay.Z, lay.bits, Options(), trace=trace)
    assert nacc.sum() == 0
    H = prep.H
    g = lay.g
    checked = 0
    for ev in trace:
        i = ev["group"]
        si = slice(i * g, (i + 1) * g)
        zx = ev["z"][:, None] + ev["x"]
        unclipped = np.all((zx >= -0.5) & (zx <= (1 << lay.bits) - 0.5), axis=1)
        C = res.Q.astype(np.float64) - np.repeat(lay.Z, g, 1)
        r = lay.W.astype(np.float64) - np.repeat(res.S, g, 1) * C
        Hr_i = r @ H[:, si]
        t = Hr_i + (res.S[:, i:i + 1] * C[:, si]) @ H[si, si]
        Rd2 = np.sum(np.diag(prep.R[i]) ** 2)
        for j in np.nonzero(unclipped)[0]:
            s = res.S[j, i]
            c = C[j, si]
            # E(q) - eta = s^2 c^T Hii c - 2 s c^T t + t^T Hii^{-1} t  (>= 0)
            best = -t[j] @ np.linalg.solve(H[si, si], t[j])
            e = s * s * c @ H[si, si] @ c - 2 * s * c @ t[j]
            assert e - best <= s * s * Rd2 / 4 * (1 + 1e-9) + 1e-12
            checked += 1
    assert checked > 10


# ---------------------------------------------------------------------------
# Format, special cases, paper-literal QR form
# ---------------------------------------------------------------------------

def test_format_preserved_and_k0_identity():
    """Sec. 3.1: bits, groups and zero points are fixed; codes stay in
    [0, 2^b - 1]. K = 0 returns the host state (Cor. host proof)."""
    lay = tiny_layer()
    prep = prepare_hessian(lay.H, lay.g)
    Z0 = lay.Z.copy()
    res = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits, Options(max_iters=3))
    assert np.array_equal(lay.Z, Z0)
    assert res.Q.min() >= 0 and res.Q.max() <= 7
    assert res.Q.shape == lay.Q0.shape and res.S.shape == lay.S0.shape
    res0 = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, lay.bits, Options(max_iters=0))
    assert np.array_equal(res0.Q, lay.Q0) and np.array_equal(res0.S, lay.S0.astype(np.float64))


def test_small_scale_groups_keep_codes():
    """App. E 'Small scales': groups with |s| <= FP32 eps get no proposal."""
    lay = small_layer(128, 8, 32, 3, seed=10)
    prep = prepare_hessian(lay.H, lay.g)
    S = lay.S0.astype(np.float64)
    S[:, 1] = FP32_EPS / 2
    Q = lay.Q0.astype(np.int64)
    trace = []
    code_sweep(prep, lay.W, S, Q, lay.Z, lay.bits, Options(), trace=trace)
    assert np.array_equal(Q[:, 32:64], lay.Q0[:, 32:64])
    assert not trace[1]["accepted"].any()


def test_canonicalization_preserves_weights():
    """App. E, Eqs. canonicalization*: the map keeps every dequantised weight
    and the codes stay in range."""
    lay = small_layer(128, 16, 32, 3, seed=12)
    rng = np.random.default_rng(0)
    S = lay.S0.astype(np.float64) * rng.choice([-1, 1], lay.S0.shape)
    S2, Q2, Z2 = canonicalize(S, lay.Q0, lay.Z, 3)
    np.testing.assert_allclose(dequantize(S2, Q2, Z2, 32), dequantize(S, lay.Q0, lay.Z, 32), rtol=1e-15)
    assert np.all(S2 >= 0) and Q2.min() >= 0 and Q2.max() <= 7 and Z2.min() >= 0 and Z2.max() <= 7


def test_group_target_equals_conditional_residual():
    """Eq. conditional_residual: A_i^T y^{(i,k)} = (H r)_i + s_i H_ii c_i
    equals A_i^T (A w - sum_{h != i} s_h A_h c_h) built from explicit A."""
    lay, X = small_layer(64, 5, 16, 3, seed=13, rank=4, tokens=300, return_X=True)
    A = X.astype(np.float64)
    H = A.T @ A
    prep = prepare_hessian(H, 16)
    C = lay.Q0.astype(np.float64) - np.repeat(lay.Z, 16, 1)
    S = lay.S0.astype(np.float64)
    r = lay.W.astype(np.float64) - np.repeat(S, 16, 1) * C
    for i in range(4):
        si = slice(i * 16, (i + 1) * 16)
        _, t = group_target(prep, r, S[:, i], C[:, si], i)
        for j in range(5):
            y = A @ lay.W[j].astype(np.float64)
            for h in range(4):
                if h != i:
                    sh = slice(h * 16, (h + 1) * 16)
                    y = y - S[j, h] * (A[:, sh] @ C[j, sh])
            np.testing.assert_allclose(t[j], A[:, si].T @ y, rtol=1e-9, atol=1e-9)


def test_h_form_matches_paper_literal_qr_form():
    """The H-form oracle and the paper-literal QR-form implementation (explicit
    A = [X; nu I], U^T Y, group QR, Eq. conditional_residual, direct group
    errors) agree on the tiny layer (16 sampled rows, K = 5, early stop on)."""
    lay, X = tiny_layer(return_X=True)
    n = X.shape[0]
    Hx = X.astype(np.float64).T @ X.astype(np.float64) / n
    damp = 0.01 * float(np.mean(np.diag(Hx)))
    prep = prepare_hessian(Hx + damp * np.eye(lay.din), lay.g)
    rows = np.arange(0, lay.dout, 16)
    # two formulations of the same float64 arithmetic: float64 scales on both
    res = refine_layer(prep, lay.W[rows], lay.S0[rows], lay.Q0[rows], lay.Z[rows], lay.bits,
                       Options(max_iters=5, fp32_scales=False))
    S3, Q3, F3 = refine_columns(X / np.sqrt(n), lay.W[rows], lay.S0[rows], lay.Q0[rows],
                                lay.Z[rows], lay.bits, lay.g, 5, nu=np.sqrt(damp),
                                fp32_scales=False)
    assert np.array_equal(Q3, res.Q)
    np.testing.assert_allclose(S3, res.S, rtol=1e-10)
    np.testing.assert_allclose(F3, res.L_final, rtol=1e-9)
    assert np.any(res.Q != lay.Q0[rows])


def test_oracle_row_independence():
    """Sec. 3.3: the objective separates over output rows, so refining a
    subset of rows gives the same result as refining the whole layer."""
    lay = small_layer(128, 24, 32, 3, seed=15)
    prep = prepare_hessian(lay.H, lay.g)
    full = refine_layer(prep, lay.W, lay.S0, lay.Q0, lay.Z, 3, Options(max_iters=4))
    rows = np.array([3, 7, 20])
    sub = refine_layer(prep, lay.W[rows], lay.S0[rows], lay.Q0[rows], lay.Z[rows], 3,
                       Options(max_iters=4))
    assert np.array_equal(sub.Q, full.Q[rows])
    np.testing.assert_allclose(sub.S, full.S[rows], rtol=1e-12)
