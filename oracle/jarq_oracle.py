"""Plain float64 CPU oracle for JARQ layer-wise refinement (H-form).

TEST INFRASTRUCTURE. This module is the slow, obviously-correct statement of
what the GPU path computes. Only the test-suite, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py`` may import it; the product path
(the C-ABI library and its Python binding) never does, and shares no code,
table or helper with it.

Notation follows the paper (JARQ: Joint Alternating Refinement for
Quantization):

* ``W`` is stored as PyTorch does, ``dout x din``; row ``j`` here is the
  paper's column ``w_j`` (Sec. 3.1, Eq. quantized_group).
* ``H = A^T A`` with ``A = [X; nu I]`` (Sec. 3.2, Eq. strict_target; App. E
  "Propagation-Corrected Targets").  For the main target ``Y = A W`` the
  objective is ``F_j = (w_j - what_j)^T H (w_j - what_j)`` (Eq.
  bbmils_columns), the QR constant being zero (App. E.1, Eq. qr_equivalence).
* The group factor ``R_i`` of the paper's thin QR ``A_i = U_i R_i`` (Eq.
  group_qr) satisfies ``R_i^T R_i = H_ii``; it is taken here as the upper
  Cholesky factor, which equals the QR factor up to row signs.  The Babai
  recursion (Eq. babai_update) is invariant to those signs.
* ``U_i^T y^{(i,k)} = R_i^{-T} A_i^T y^{(i,k)}`` and
  ``A_i^T y^{(i,k)} = (H r)_i + H_ii (s_i c_i)`` with ``r = w - what`` (Eq.
  conditional_residual), so ``v = R_i^{-T}[(H r)_i + s_i H_ii c_i] / s_i``.

Readings of the paper that this oracle takes where the text is silent:

1. Iteration k = refit S for Q^{(k-1)}, then one Gauss-Seidel Babai sweep on
   S^{(k)} (Sec. 3.3).  No extra refit after the K-th sweep.
2. ``round`` is round-half-to-even of ``z + x`` (numpy ``rint``).
3. The ridge test uses the exact float64 spectrum (App. E "Solving for
   scales"); a failed retry marks the row NUMERICAL and keeps its last
   state.
4. Acceptance compares the change of the group objective, ``dF < 0``
   (Sec. 3.3.2; App. E "Small scales"); proposals equal to the current codes
   give ``dF == 0`` and are not accepted.
5. The small-scale test is ``|s| > FLT_EPSILON`` (absolute).
6. Early stop (Eq. strict_stopping) is tested for k >= 2 right after the
   scale update, using the full objective L^{(k)}; the new scales are kept.
7. The scales are single-precision numbers: App. E states that the scale
   system is solved in FP32, and the scale table the refinement updates is
   an FP32 array.  The oracle solves in float64 and stores the correctly
   rounded float32 value after every solve (``Options.fp32_scales``); the
   objective, the Babai recursion and the acceptance test then run in
   float64 on those float32 scales.  ``fp32_scales=False`` keeps float64
   scales, for the paper's exact worked examples.
8. ``Options.ridge_accept`` (off by default, as in the paper's runs) keeps a
   ridge-stabilised solve only when it does not increase F_j, and the
   previous scales otherwise (App. G, Remark ridge-acceptance).

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
against the paper's worked examples (App. G, Props. grid-staleness and
multicode-descent), closed forms, brute force and invariants.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import scipy.linalg

# FP32 machine epsilon, the paper's eps_fp (App. E "Solving for scales").
FP32_EPS = float(np.finfo(np.float32).eps)

# Per-row status codes (same numbering as the C-ABI's status enum).
ROW_OK = 0
ROW_NUMERICAL = 3


@dataclasses.dataclass
class Options:
    """Solver settings (App. E "Numerical Updates and Stopping")."""

    max_iters: int = 3          # K (Sec. 3.3, "all main experiments use K=3")
    tau: float = 1e-5           # Eq. strict_stopping
    early_stop: bool = True
    ridge: float = 1e-4         # lambda of the stabilised scale solve
    rcond: float = 1e-10        # spectrum test threshold
    eps: float = FP32_EPS       # eps_fp
    fp32_scales: bool = True    # store each solved scale as float32 (reading 7)
    ridge_accept: bool = False  # Remark ridge-acceptance: keep a ridge solve only if F does not rise


@dataclasses.dataclass
class Prepared:
    """Symmetrised Hessian and its per-group upper Cholesky factors."""

    H: np.ndarray               # float64 [d][d]
    R: list                     # G arrays, float64 [g][g], upper, H_ii = R^T R
    g: int

    @property
    def d(self) -> int:
        return self.H.shape[0]

    @property
    def G(self) -> int:
        return self.d // self.g


class NotSPD(ValueError):
    """A diagonal block H_ii is not positive definite (Eq. group_qr needs it)."""


def prepare_hessian(H, g: int, nu2: float = 0.0) -> Prepared:
    """Symmetrise ``H`` (+ ``nu2 I``) and factor each diagonal block.

    Sec. 3.3.2, Eq. group_qr: the group factors are precomputed once and
    reused for every output row and iteration.  ``nu2`` adds the paper's
    ``nu^2 I`` (Eq. strict_target) when ``H`` was built without it.
    """
    H = np.asarray(H, dtype=np.float64)
    d = H.shape[0]
    if H.shape != (d, d) or d % g != 0:
        raise ValueError("H must be square with din divisible by the group size")
    Hs = 0.5 * (H + H.T)
    if nu2:
        Hs = Hs + nu2 * np.eye(d)
    R = []
    for i in range(d // g):
        blk = Hs[i * g:(i + 1) * g, i * g:(i + 1) * g]
        try:
            Lc = np.linalg.cholesky(blk)
        except np.linalg.LinAlgError as e:
            raise NotSPD(f"H block {i} is not positive definite") from e
        R.append(Lc.T.copy())
    return Prepared(H=Hs, R=R, g=g)


def dequantize(S, Q, Z, g: int):
    """``what_j = D_{s_j}(q_j - z_j)`` (Sec. 3.1, Eq. quantized_group)."""
    S = np.asarray(S, dtype=np.float64)
    C = np.asarray(Q, dtype=np.float64) - np.repeat(np.asarray(Z, dtype=np.float64), g, axis=1)
    return np.repeat(S, g, axis=1) * C


def objective(prep: Prepared, W, S, Q, Z):
    """Per-row objective ``F_j = r_j^T H r_j``, ``r_j = w_j - what_j``.

    Sec. 3.2, Eq. bbmils_columns, for the main target ``Y = A W``.
    """
    R = np.asarray(W, dtype=np.float64) - dequantize(S, Q, Z, prep.g)
    return np.einsum("jd,jd->j", R @ prep.H, R)


def scale_system(prep: Prepared, W, Q, Z):
    """Normal equations of the joint scale fit for each row.

    Sec. 3.3.1, Eqs. scale_design and scale_normal_equations:
    ``Gram_j[i,h] = (A_i c_i)^T (A_h c_h) = c_i^T H_ih c_h`` and
    ``rhs_j[i] = (A_i c_i)^T y_j = c_i^T (H w_j)_i``.
    """
    g, G, H = prep.g, prep.G, prep.H
    W = np.asarray(W, dtype=np.float64)
    C = np.asarray(Q, dtype=np.float64) - np.repeat(np.asarray(Z, dtype=np.float64), g, axis=1)
    rows = W.shape[0]
    HW = W @ H
    Gram = np.empty((rows, G, G))
    rhs = np.empty((rows, G))
    for h in range(G):
        sh = slice(h * g, (h + 1) * g)
        HCh = C[:, sh] @ H[sh, :]            # row j: (H c_h)^T over all d
        for i in range(G):
            si = slice(i * g, (i + 1) * g)
            Gram[:, i, h] = np.einsum("jk,jk->j", C[:, si], HCh[:, si])
    for i in range(G):
        si = slice(i * g, (i + 1) * g)
        rhs[:, i] = np.einsum("jk,jk->j", C[:, si], HW[:, si])
    return Gram, rhs


def solve_scales(Gram, rhs, opt: Options):
    """Stabilised Cholesky solve of one row's G x G system.

    App. E "Solving for scales": symmetrise; if the spectrum is nonfinite,
    ``lambda_min <= rcond * max(|lambda_max|, eps)`` or Cholesky fails, add
    ``ridge * I`` and factor again; if that fails, report a numerical error.
    Returns ``(s, ridge_used, ok)``.
    """
    Gm = 0.5 * (Gram + Gram.T)
    need_ridge = False
    if not np.all(np.isfinite(Gm)):
        need_ridge = True
    else:
        lam = np.linalg.eigvalsh(Gm)
        if lam[0] <= opt.rcond * max(abs(lam[-1]), opt.eps):
            need_ridge = True
    if not need_ridge:
        try:
            Lc = np.linalg.cholesky(Gm)
        except np.linalg.LinAlgError:
            need_ridge = True
    if need_ridge:
        Gm = Gm + opt.ridge * np.eye(Gm.shape[0])
        try:
            Lc = np.linalg.cholesky(Gm)
        except np.linalg.LinAlgError:
            return None, True, False
        if not np.all(np.isfinite(Lc)):
            return None, True, False
    y = scipy.linalg.solve_triangular(Lc, rhs, lower=True)
    s = scipy.linalg.solve_triangular(Lc.T, y, lower=False)
    if not np.all(np.isfinite(s)):
        return None, need_ridge, False
    return s, need_ridge, True


def babai_proposal(R_i, v, z, qmax):
    """Bounded Babai nearest-plane proposal for one group, all rows at once.

    Sec. 3.3.2, Eq. babai_update: for ``l = g..1``,
    ``q_l = clip(round(z + (v_l - sum_{h>l} R_lh (q_h - z)) / R_ll))``.
    ``v``: [rows][g]; ``z``: [rows].  Returns ``(q, x)`` where ``x`` holds the
    pre-round values ``(v_l - sum ...)/R_ll`` (the paper's worked examples
    print ``z + x``).
    """
    rows, g = v.shape
    q = np.zeros((rows, g))
    x = np.zeros((rows, g))
    zc = z[:, None]
    for l in range(g - 1, -1, -1):
        acc = v[:, l] - (q[:, l + 1:] - zc) @ R_i[l, l + 1:]
        x[:, l] = acc / R_i[l, l]
        q[:, l] = np.clip(np.rint(z + x[:, l]), 0, qmax)
    return q, x


def group_target(prep: Prepared, r, S_i, C_i, i):
    """``A_i^T y^{(i,k)} = (H r)_i + s_i H_ii c_i`` (Eq. conditional_residual).

    ``r`` holds the current residual ``w - what`` (new codes for groups
    before ``i``, previous codes for the rest).  Returns ``(Hr_i, t)``.
    """
    g, H = prep.g, prep.H
    si = slice(i * g, (i + 1) * g)
    Hr_i = r @ H[:, si]
    t = Hr_i + (S_i[:, None] * C_i) @ H[si, si]
    return Hr_i, t


def code_sweep(prep: Prepared, W, S, Q, Z, bits, opt: Options, rows=None,
               trace=None):
    """One Gauss-Seidel sweep of bounded Babai proposals over the groups.

    Sec. 3.3.2 (Eqs. conditional_residual, group_bils, group_qr,
    babai_update) and App. E "Small scales".  Modifies ``Q`` in place for
    the given ``rows`` and returns the per-row sum of accepted objective
    changes and the per-row count of accepted proposals.
    """
    g, G, H = prep.g, prep.G, prep.H
    qmax = (1 << bits) - 1
    if rows is None:
        rows = np.arange(Q.shape[0])
    Wr = np.asarray(W, dtype=np.float64)[rows]
    Sr = np.asarray(S, dtype=np.float64)[rows]
    Zr = np.asarray(Z, dtype=np.float64)[rows]
    Qr = np.asarray(Q, dtype=np.float64)[rows].copy()
    dF_sum = np.zeros(len(rows))
    n_acc = np.zeros(len(rows), dtype=np.int64)
    for i in range(G):
        si = slice(i * g, (i + 1) * g)
        C = Qr - np.repeat(Zr, g, axis=1)
        r = Wr - np.repeat(Sr, g, axis=1) * C
        s_i = Sr[:, i]
        Hr_i, t = group_target(prep, r, s_i, C[:, si], i)
        live = np.abs(s_i) > opt.eps
        s_safe = np.where(live, s_i, 1.0)
        # v = U_i^T y / s = R_i^{-T} A_i^T y / s   (Eq. babai_update)
        v = scipy.linalg.solve_triangular(prep.R[i], t.T, trans="T", lower=False).T / s_safe[:, None]
        qc, x = babai_proposal(prep.R[i], v, Zr[:, i], qmax)
        delta = s_i[:, None] * (qc - Qr[:, si])
        dF = -2.0 * np.einsum("jk,jk->j", delta, Hr_i) + np.einsum("jk,jk->j", delta @ H[si, si], delta)
        with np.errstate(invalid="ignore"):
            accept = live & np.isfinite(dF) & (dF < 0.0)
        Qr[accept, si] = qc[accept]
        dF_sum[accept] += dF[accept]
        n_acc += accept
        if trace is not None:
            trace.append(dict(kind="babai", group=i, s=s_i.copy(), x=x.copy(),
                              z=Zr[:, i].copy(), proposal=qc.copy(), dF=dF.copy(),
                              accepted=accept.copy(), live=live.copy()))
    Q[rows] = Qr.astype(Q.dtype)
    return dF_sum, n_acc


@dataclasses.dataclass
class Result:
    S: np.ndarray
    Q: np.ndarray
    L_host: np.ndarray
    L_final: np.ndarray
    iters: np.ndarray
    accepted: np.ndarray
    ridge_hits: np.ndarray
    row_status: np.ndarray
    L_hist: list                # L^{(k)} after each scale update, per row (NaN if stopped)


def refine_layer(prep: Prepared, W, S0, Q0, Z, bits: int, opt: Options = None,
                 trace=None, const=None) -> Result:
    """JARQ's alternating refinement of one layer (Sec. 3.3; App. E).

    For ``k = 1..K`` each active row (i) refits all G scales jointly for its
    current codes (Sec. 3.3.1), computes ``L^{(k)}`` and applies the early
    stop of Eq. strict_stopping for ``k >= 2``, then (ii) runs one bounded
    Babai sweep over its groups on the new scales (Sec. 3.3.2).  Rows are
    independent (Sec. 3.3, "separates over output columns").

    ``const`` (optional, per row) is a constant added to every objective
    value L: a target outside the range of A contributes the orthogonal
    residual c_j, which Algorithm 1 carries in its objective (App.
    "Propagation-Corrected Targets and QEP"); it moves the early-stop test and
    the reported L, never a scale or a code.
    """
    opt = opt or Options()
    W = np.asarray(W, dtype=np.float64)
    S = np.array(S0, dtype=np.float64, copy=True)
    Q = np.array(Q0, dtype=np.int64, copy=True)
    Z = np.asarray(Z)
    p = W.shape[0]
    if Q.min(initial=0) < 0 or Q.max(initial=0) > (1 << bits) - 1:
        raise ValueError("codes outside the b-bit range")
    c = np.zeros(p) if const is None else np.asarray(const, dtype=np.float64)
    L_host = objective(prep, W, S, Q, Z) + c
    active = np.ones(p, dtype=bool)
    iters = np.zeros(p, dtype=np.int64)
    accepted = np.zeros(p, dtype=np.int64)
    ridge_hits = np.zeros(p, dtype=np.int64)
    status = np.zeros(p, dtype=np.int64)
    L_prev = np.full(p, np.nan)
    L_hist = []
    for k in range(1, opt.max_iters + 1):
        rows = np.nonzero(active)[0]
        if rows.size == 0:
            break
        Gram, rhs = scale_system(prep, W[rows], Q[rows], Z[rows])
        for n, j in enumerate(rows):
            s, used_ridge, ok = solve_scales(Gram[n], rhs[n], opt)
            ridge_hits[j] += int(used_ridge)
            if not ok:
                status[j] = ROW_NUMERICAL
                active[j] = False
                continue
            s_old = S[j].copy()
            S[j] = s.astype(np.float32) if opt.fp32_scales else s
            if used_ridge and opt.ridge_accept:
                # Remark ridge-acceptance: the ridge solution is kept only when
                # it does not increase F_j; otherwise the previous scales stay
                F_new = objective(prep, W[j:j + 1], S[j:j + 1], Q[j:j + 1], Z[j:j + 1])[0]
                F_old = objective(prep, W[j:j + 1], s_old[None], Q[j:j + 1], Z[j:j + 1])[0]
                if not F_new <= F_old:
                    S[j] = s_old
        rows = np.nonzero(active)[0]
        iters[rows] = k
        L = np.full(p, np.nan)
        L[rows] = objective(prep, W[rows], S[rows], Q[rows], Z[rows]) + c[rows]
        L_hist.append(L.copy())
        if trace is not None:
            trace.append(dict(kind="scale", k=k, rows=rows.copy(), S=S[rows].copy(), L=L[rows].copy()))
        if opt.early_stop and k >= 2:
            dec = L_prev[rows] - L[rows]
            stop = (dec / np.maximum(np.abs(L_prev[rows]), opt.eps) <= opt.tau) | (np.abs(dec) <= opt.tau)
            active[rows[stop]] = False
            rows = rows[~stop]
        L_prev = L
        if rows.size == 0:
            break
        _, n_acc = code_sweep(prep, W, S, Q, Z, bits, opt, rows=rows, trace=trace)
        accepted[rows] += n_acc
        if trace is not None:
            trace.append(dict(kind="sweep", k=k, rows=rows.copy(),
                              F=objective(prep, W[rows], S[rows], Q[rows], Z[rows])))
    L_final = objective(prep, W, S, Q, Z) + c
    return Result(S=S, Q=Q, L_host=L_host, L_final=L_final, iters=iters,
                  accepted=accepted, ridge_hits=ridge_hits, row_status=status,
                  L_hist=L_hist)


def canonicalize(S, Q, Z, bits):
    """Map negative scales to the equivalent positive form.

    App. E "Representing Negative Scales", Eq. canonicalization:
    ``s' = -s, q' = qmax - q, z' = qmax - z`` for every group with ``s < 0``.
    """
    qmax = (1 << bits) - 1
    S = np.array(S, dtype=np.float64, copy=True)
    Q = np.array(Q, copy=True)
    Z = np.array(Z, copy=True)
    g = Q.shape[1] // S.shape[1]
    neg = S < 0
    S[neg] = -S[neg]
    Z[neg] = qmax - Z[neg]
    negx = np.repeat(neg, g, axis=1)
    Q[negx] = qmax - Q[negx]
    return S, Q, Z
