"""Paper-literal QR-form oracle for tiny JARQ problems.

TEST INFRASTRUCTURE, like ``jarq_oracle``.  It exists to pin the H-form
oracle: it never forms ``H`` but works with the augmented design matrix
``A = [X; nu I]`` and target ``Y`` exactly as the paper writes them, one
output column at a time, in float64:

* Sec. 3.2, Eq. strict_target: ``A = [X; nu I]``, ``Y = [Y*; nu W]``.
* Sec. 3.3 "Layerwise procedure" and App. E.1, Eq. qr_equivalence: thin QR
  ``A = U R``, reduced target ``Ybar = U^T Y``; the objective is
  ``||Ybar - R What||^2`` plus the constant ``||(I - U U^T) Y||^2``.
* Sec. 3.3.1, Eqs. scale_design / scale_normal_equations on the reduced
  design ``R = [R_1 .. R_G]`` (column blocks).
* Sec. 3.3.2, Eq. conditional_residual (the target with the latest codes of
  the other groups subtracted), Eq. group_qr (thin QR of each reduced column
  block ``R_{:,i} = U_i R_i`` with numpy's arbitrary row signs), Eq.
  babai_update, and acceptance on the group error of Eq. group_bils
  evaluated directly.
* App. E "Early stopping", Eq. strict_stopping, on the full objective
  including the QR constant.

Only for tiny inputs: plain Python loops over columns, groups and
coordinates.
"""
from __future__ import annotations

import numpy as np

FP32_EPS = float(np.finfo(np.float32).eps)


def refine_columns(X, W, S0, Q0, Z, bits, g, K, nu=0.0, Ystar=None, tau=1e-5,
                   early_stop=True, ridge=1e-4, rcond=1e-10, eps=FP32_EPS,
                   fp32_scales=True):
    """Refine every output column of a tiny layer with the paper's QR form.

    ``X``: n x din calibration inputs; ``W``: dout x din (row j = paper's
    column w_j); ``Ystar``: n x dout activation target (default ``X W^T``,
    the main target of Sec. 3.2).  ``fp32_scales`` stores every solved scale
    as float32, the single-precision scale solve of App. E.  Returns
    ``(S, Q, F_final)``.
    """
    X = np.asarray(X, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    n, d = X.shape
    p = W.shape[0]
    G = d // g
    qmax = (1 << bits) - 1
    A = np.vstack([X, nu * np.eye(d)]) if nu else X.copy()
    if Ystar is None:
        Ystar = X @ W.T
    Y = np.vstack([Ystar, nu * W.T]) if nu else np.asarray(Ystar, dtype=np.float64)
    U, R = np.linalg.qr(A, mode="reduced")
    Ybar = U.T @ Y
    const = np.sum((Y - U @ Ybar) ** 2, axis=0)
    blocks = [R[:, i * g:(i + 1) * g] for i in range(G)]
    gqr = [np.linalg.qr(B, mode="reduced") for B in blocks]
    S = np.array(S0, dtype=np.float64, copy=True)
    Q = np.array(Q0, dtype=np.int64, copy=True)
    F_final = np.zeros(p)
    for j in range(p):
        s = S[j].copy()
        q = Q[j].astype(np.float64)
        z = np.asarray(Z[j], dtype=np.float64)
        ybar = Ybar[:, j]

        def full_obj(s_, q_):
            what = np.repeat(s_, g) * (q_ - np.repeat(z, g))
            return float(np.sum((ybar - R @ what) ** 2) + const[j])

        L_prev = None
        for k in range(1, K + 1):
            B = np.stack([blocks[i] @ (q[i * g:(i + 1) * g] - z[i]) for i in range(G)], axis=1)
            Gm = B.T @ B
            Gm = 0.5 * (Gm + Gm.T)
            rhs = B.T @ ybar
            lam = np.linalg.eigvalsh(Gm) if np.all(np.isfinite(Gm)) else None
            bad = lam is None or lam[0] <= rcond * max(abs(lam[-1]), eps)
            try:
                if bad:
                    raise np.linalg.LinAlgError
                s_new = np.linalg.solve(np.linalg.cholesky(Gm).T, np.linalg.solve(np.linalg.cholesky(Gm), rhs))
            except np.linalg.LinAlgError:
                Lc = np.linalg.cholesky(Gm + ridge * np.eye(G))
                s_new = np.linalg.solve(Lc.T, np.linalg.solve(Lc, rhs))
            s = s_new.astype(np.float32).astype(np.float64) if fp32_scales else s_new
            L = full_obj(s, q)
            if early_stop and k >= 2:
                dec = L_prev - L
                if dec / max(abs(L_prev), eps) <= tau or abs(dec) <= tau:
                    break
            L_prev = L
            for i in range(G):
                if abs(s[i]) <= eps:
                    continue
                # Eq. conditional_residual: subtract the latest contributions of
                # every other group (new codes for g < i, old ones for g > i).
                y_ik = ybar.copy()
                for h in range(G):
                    if h != i:
                        y_ik -= s[h] * (blocks[h] @ (q[h * g:(h + 1) * g] - z[h]))
                Ui, Ri = gqr[i]
                v = Ui.T @ y_ik / s[i]
                cand = np.zeros(g)
                for l in range(g - 1, -1, -1):
                    acc = v[l] - sum(Ri[l, hh] * (cand[hh] - z[i]) for hh in range(l + 1, g))
                    cand[l] = min(max(np.rint(z[i] + acc / Ri[l, l]), 0), qmax)
                old = q[i * g:(i + 1) * g]
                E_new = np.sum((y_ik - s[i] * blocks[i] @ (cand - z[i])) ** 2)
                E_old = np.sum((y_ik - s[i] * blocks[i] @ (old - z[i])) ** 2)
                if np.isfinite(E_new) and E_new < E_old:
                    q[i * g:(i + 1) * g] = cand
        S[j] = s
        Q[j] = q.astype(np.int64)
        F_final[j] = full_obj(s, q)
    return S, Q, F_final
