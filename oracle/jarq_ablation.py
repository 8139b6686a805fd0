"""Mechanism ablations of JARQ (test infrastructure, like jarq_oracle).

TEST INFRASTRUCTURE: only the test-suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this module.

App. "Refinement Mechanisms" (Tab. mechanism-summary (a)) isolates the
ingredients of JARQ on fixed layers:

* scale fits with the codes fixed (App. "Joint Scale Fitting"):
  - independent: each group's scale fitted to that group's own
    contribution, s~_i = b_i^T A_i w_i / ||b_i||^2 with b_i = A_i c_i
    (Eq. independent-fit), i.e. c_i^T H_ii w_i / c_i^T H_ii c_i;
  - coordinate descent: one scale at a time against the full residual,
    each update the exact minimiser along that coordinate,
    s_i <- s_i + c_i^T (H r)_i / c_i^T H_ii c_i, groups in order, a fixed
    number of passes (three in the table);
  - joint: the normal equations of Eq. scale_normal_equations;
  the gap of a method is 100 (L_method - L_joint) / L_base with L_base the
  objective before the fit;
* multi-code updates (App. "Multi-Code Updates"): for one output row and
  one group, with the scales and the other groups fixed, single-code
  updates until no one-code change strictly lowers the objective, then one
  Babai proposal from that state (Eq. babai_update), accepted iff it
  strictly lowers the objective;
* fixed grid versus joint (App. "Fixed-Grid versus Joint Refinement"):
  Fixed keeps the host scales and only runs code sweeps.

Readings (the paper leaves these open): a group whose c_i^T H_ii c_i is 0
keeps its scale in the independent and coordinate-descent fits (every
scale gives the same objective there); the single-code search visits the
coordinates in order, moves each to its best code when that strictly
lowers the objective, and repeats full passes until a pass moves nothing;
all these fits return float64 scales rounded to float32 at the end, like
the joint solve (reading of the FP32 scale table).
"""
from __future__ import annotations

import numpy as np
import scipy.linalg

from .jarq_oracle import (Options, babai_proposal, objective, refine_layer, scale_system,
                          solve_scales)


def _codes(Q, Z, g):
    return np.asarray(Q, dtype=np.float64) - np.repeat(np.asarray(Z, dtype=np.float64), g, axis=1)


def independent_scales(prep, W, S0, Q, Z):
    """Eq. independent-fit for every row and group (float64)."""
    g, G, H = prep.g, prep.G, prep.H
    W = np.asarray(W, dtype=np.float64)
    C = _codes(Q, Z, g)
    S = np.array(S0, dtype=np.float64, copy=True)
    for i in range(G):
        si = slice(i * g, (i + 1) * g)
        Hii = H[si, si]
        num = np.einsum("jk,jk->j", C[:, si] @ Hii, W[:, si])
        den = np.einsum("jk,jk->j", C[:, si] @ Hii, C[:, si])
        ok = den > 0
        S[ok, i] = num[ok] / den[ok]
    return S


def coordinate_descent_scales(prep, W, S0, Q, Z, passes: int = 3):
    """Cyclic exact coordinate minimisation of F over the scales (float64),
    starting from S0, on the Gram system of Eq. scale_normal_equations."""
    Gram, rhs = scale_system(prep, W, Q, Z)
    S = np.array(S0, dtype=np.float64, copy=True)
    for j in range(S.shape[0]):
        s = S[j]
        grad = rhs[j] - Gram[j] @ s            # c_i^T (H r)_i for every group
        for _ in range(passes):
            for i in range(s.size):
                d = Gram[j, i, i]
                if d > 0:
                    step = grad[i] / d
                    s[i] += step
                    grad -= Gram[j, :, i] * step
        S[j] = s
    return S


def joint_scales(prep, W, S0, Q, Z, opt: Options = None):
    """The joint least-squares fit (Sec. 3.3.1) of every row; rows whose
    system fails keep S0."""
    opt = opt or Options()
    Gram, rhs = scale_system(prep, W, Q, Z)
    S = np.array(S0, dtype=np.float64, copy=True)
    for j in range(S.shape[0]):
        s, _, ok = solve_scales(Gram[j], rhs[j], opt)
        if ok:
            S[j] = s
    return S


def scale_fit_gaps(prep, W, S0, Q, Z, passes: int = 3):
    """Objectives of the three fits (float32 scales) and the gaps of
    Tab. mechanism-summary: 100 (L_method - L_joint) / L_base."""
    L_base = objective(prep, W, S0, Q, Z)
    fits = {"joint": joint_scales(prep, W, S0, Q, Z),
            "independent": independent_scales(prep, W, S0, Q, Z),
            "coordinate": coordinate_descent_scales(prep, W, S0, Q, Z, passes)}
    out = {"L_base": L_base}
    for k, S in fits.items():
        S32 = S.astype(np.float32)
        out["S_" + k] = S32
        out["L_" + k] = objective(prep, W, S32, Q, Z)
    for k in ("independent", "coordinate"):
        out["gap_" + k] = 100.0 * (out["L_" + k] - out["L_joint"]) / L_base
    return out


def single_code_search(Hii, hr, s: float, q, z: float, qmax: int):
    """Single-code updates of one group with its scale and the other groups
    fixed, until no one-code change strictly lowers the objective.

    ``Hii`` the g x g block, ``hr`` = (H r)_i for the current residual,
    ``q`` the group's codes.  Changing code l by one step Delta = s (q' - q_l)
    of the dequantised weight changes F by -2 Delta (H r)_l + Delta^2 H_ll
    (r loses Delta in coordinate l), after which (H r)_i loses Delta H_ii[:, l].
    Returns (codes, (H r)_i, number of moves)."""
    q = np.array(q, dtype=np.float64, copy=True)
    hr = np.array(hr, dtype=np.float64, copy=True)
    g = q.size
    cand = np.arange(qmax + 1, dtype=np.float64)
    moves = 0
    while True:
        moved = False
        for l in range(g):
            delta = s * (cand - q[l])
            dF = -2.0 * delta * hr[l] + delta * delta * Hii[l, l]
            k = int(np.argmin(dF))
            if dF[k] < 0.0:
                hr -= delta[k] * Hii[:, l]
                q[l] = cand[k]
                moved = True
                moves += 1
        if not moved:
            return q, hr, moves


def is_single_code_stationary(Hii, hr, s: float, q, qmax: int) -> bool:
    """The float64 check: no allowed code of any coordinate strictly lowers F."""
    cand = np.arange(qmax + 1, dtype=np.float64)
    for l in range(q.size):
        delta = s * (cand - q[l])
        if np.any(-2.0 * delta * hr[l] + delta * delta * Hii[l, l] < 0.0):
            return False
    return True


def multicode_probe(prep, W, S, Q, Z, bits: int, i: int, eps: float = np.finfo(np.float32).eps):
    """App. "Multi-Code Updates" for group i of every row: single-code
    search, then one Babai proposal from the stationary state.

    Returns a dict of per-row arrays: ``q_search`` (codes after the search),
    ``moves``, ``accepted`` (the proposal strictly lowers F), ``changed``
    (codes the proposal changes), ``dF`` (its change of F).  Rows whose
    |s_i| <= eps are skipped (App. E "Small scales": accepted False)."""
    g, H = prep.g, prep.H
    qmax = (1 << bits) - 1
    si = slice(i * g, (i + 1) * g)
    W = np.asarray(W, dtype=np.float64)
    S = np.asarray(S, dtype=np.float64)
    Zf = np.asarray(Z, dtype=np.float64)
    C = _codes(Q, Z, g)
    R = W - np.repeat(S, g, axis=1) * C
    Hii = H[si, si]
    Ri = prep.R[i]
    p = W.shape[0]
    out = {"q_search": np.array(Q, dtype=np.float64)[:, si].copy(),
           "moves": np.zeros(p, np.int64), "accepted": np.zeros(p, bool),
           "changed": np.zeros(p, np.int64), "dF": np.zeros(p)}
    for j in range(p):
        s = S[j, i]
        if not abs(s) > eps:
            continue
        hr = R[j] @ H[:, si]
        q0 = np.asarray(Q, dtype=np.float64)[j, si]
        q, hr, moves = single_code_search(Hii, hr, s, q0, Zf[j, i], qmax)
        out["q_search"][j] = q
        out["moves"][j] = moves
        # Babai target from the searched state (Eq. conditional_residual):
        # A_i^T y = (H r)_i + s H_ii c_i, v = R_i^{-T} A_i^T y / s
        c = q - Zf[j, i]
        t = hr + s * (Hii @ c)
        v = scipy.linalg.solve_triangular(Ri, t, trans="T", lower=False) / s
        qb, _ = babai_proposal(Ri, v[None, :], np.array([Zf[j, i]]), qmax)
        qb = qb[0]
        delta = s * (qb - q)
        dF = -2.0 * delta @ hr + delta @ Hii @ delta
        out["dF"][j] = dF
        out["accepted"][j] = bool(np.isfinite(dF) and dF < 0.0)
        out["changed"][j] = int(np.sum(qb != q))
    return out


def refine_fixed_grid(prep, W, S0, Q0, Z, bits: int, sweeps: int, opt: Options = None):
    """Fixed: the host scales stay, ``sweeps`` Babai sweeps over the groups
    (Sec. 3.3.2) update the codes; returns (Q, objective after each sweep)."""
    from .jarq_oracle import code_sweep
    opt = opt or Options()
    Q = np.array(Q0, dtype=np.int64, copy=True)
    S = np.asarray(S0, dtype=np.float64)
    hist = []
    for _ in range(sweeps):
        code_sweep(prep, W, S, Q, Z, bits, opt)
        hist.append(objective(prep, W, S, Q, Z))
    return Q, hist


def refine_joint(prep, W, S0, Q0, Z, bits: int, iters: int):
    """Joint: the JARQ loop (Algorithm 1) for ``iters`` iterations, early stop off."""
    return refine_layer(prep, W, S0, Q0, Z, bits, Options(max_iters=iters, early_stop=False))
