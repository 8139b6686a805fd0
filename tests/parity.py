"""Helpers comparing the CUDA path with the oracle (test infrastructure).

Codes are integers decided by floating point, so trajectories of the GPU
and the float64 oracle may part at a rounding or acceptance near-tie; after
that both are valid descent paths.  ``lockstep`` therefore steps both sides
one iteration at a time from the oracle's state and requires every
difference to start at a near-tie of the oracle's own values.
"""
from __future__ import annotations

import numpy as np

from oracle import Options, objective, prepare_hessian, refine_layer

TOL_ROUND = 1e-3      # |frac(z + x) - 1/2| below this is a rounding near-tie
TOL_ACCEPT = 1e-6     # |dF| / F_row below this is an acceptance near-tie
TOL_STOP = 1e-6       # |dL/L - tau| below this is an early-stop near-tie


def gpu_refine(lay, K, early_stop=False, device="cuda", S=None, Q=None, host=False,
               **opt):
    """Run jarq_refine_layer on a layer; returns numpy (S, Q, stats)."""
    import torch
    from paper_2609_38599_gb300 import jarq
    S0 = lay.S0 if S is None else S
    Q0 = lay.Q0 if Q is None else Q
    if host:
        H = np.ascontiguousarray(lay.H, dtype=np.float32)
        hess = jarq.prepare(H, lay.g)
        Sx = np.array(S0, dtype=np.float32, copy=True)
        Qx = np.array(Q0, dtype=np.uint8, copy=True)
        st = jarq.refine(hess, np.ascontiguousarray(lay.W, dtype=np.float32), Sx, Qx,
                         np.ascontiguousarray(lay.Z, dtype=np.int32), lay.bits,
                         max_iters=K, early_stop=int(early_stop), raise_on_error=False, **opt)
        hess.close()
        return Sx, Qx, st
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=device, dtype=dt).contiguous()
    hess = jarq.prepare(t(lay.H, torch.float32), lay.g)
    W = t(lay.W, torch.float32)
    Sx = t(S0, torch.float32)
    Qx = t(Q0, torch.uint8)
    Z = t(lay.Z, torch.int32)
    st = jarq.refine(hess, W, Sx, Qx, Z, lay.bits, max_iters=K, early_stop=int(early_stop),
                     raise_on_error=False, **opt)
    torch.cuda.synchronize()
    out = (Sx.cpu().numpy(), Qx.cpu().numpy(),
           {k: getattr(st, k).cpu().numpy() for k in
            ("L_host", "L_final", "iters", "accepted", "ridge_hits", "row_status")})
    out[2]["status"] = st.status
    hess.close()
    return out


def compare_final(lay, prep, res, S_gpu, Q_gpu, stats):
    """Final-state comparison; returns a dict of parity figures."""
    same_rows = np.all(Q_gpu == res.Q, axis=1)
    rel_S = np.abs(S_gpu - res.S) / np.maximum(np.abs(res.S), 1e-30)
    F_gpu_state = objective(prep, lay.W, S_gpu, Q_gpu, lay.Z)   # oracle on the GPU's state
    out = dict(
        codes_same=float(np.mean(Q_gpu == res.Q)),
        rows_same=float(np.mean(same_rows)),
        S_rel_max_same_rows=float(rel_S[same_rows].max()) if same_rows.any() else 0.0,
        F_rel_max_same_rows=float(np.max(np.abs(F_gpu_state[same_rows] - res.L_final[same_rows])
                                         / np.abs(res.L_final[same_rows]))) if same_rows.any() else 0.0,
        F_rel_all=float(np.max(np.abs(F_gpu_state - res.L_final) / np.abs(res.L_final))),
        Lfinal_vs_oracle_state=float(np.max(np.abs(stats["L_final"] - F_gpu_state) / np.abs(F_gpu_state))),
        Lhost_rel=float(np.max(np.abs(stats["L_host"] - res.L_host) / np.abs(res.L_host))),
        gpu_no_worse_than_host=bool(np.all(F_gpu_state <= res.L_host * (1 + 1e-5))),
        sum_ratio=float(F_gpu_state.sum() / res.L_final.sum()),
    )
    return out


def _round_tie(zx, qmax):
    frac = zx - np.floor(zx)
    near_half = np.abs(frac - 0.5) < TOL_ROUND
    near_clip = (np.abs(zx + 0.5) < TOL_ROUND) | (np.abs(zx - (qmax + 0.5)) < TOL_ROUND)
    return near_half | near_clip


def lockstep(lay, K, gpu_step, early_stop=False, tau=1e-5):
    """Step GPU and oracle one iteration at a time from the oracle's state.

    ``gpu_step(S, Q)`` runs one GPU iteration from (S, Q) and returns numpy
    (S, Q).  Returns per-iteration records; raises AssertionError on a
    difference that does not start at a near-tie.
    """
    prep = prepare_hessian(lay.H, lay.g)
    g, qmax = lay.g, (1 << lay.bits) - 1
    S = np.array(lay.S0, dtype=np.float64)
    Q = np.array(lay.Q0, dtype=np.int64)
    records = []
    for k in range(1, K + 1):
        trace = []
        res = refine_layer(prep, lay.W, S, Q, lay.Z, lay.bits,
                           Options(max_iters=1, early_stop=False), trace=trace)
        Sg, Qg = gpu_step(S.astype(np.float32), Q.astype(np.uint8))
        rel_S = float(np.max(np.abs(Sg - res.S) / np.maximum(np.abs(res.S), 1e-30)))
        assert rel_S < 1e-4, f"iteration {k}: scales differ by {rel_S}"
        babai = [ev for ev in trace if ev["kind"] == "babai"]
        bad_rows = np.nonzero(np.any(Qg != res.Q, axis=1))[0]
        F_row = res.L_final
        unexplained = []
        for j in bad_rows:
            i = int(np.nonzero(np.any((Qg[j] != res.Q[j]).reshape(-1, g), axis=1))[0][0])
            ev = babai[i]
            zx = ev["z"][j] + ev["x"][j]
            ties = _round_tie(zx, qmax)
            acc_tie = abs(ev["dF"][j]) <= TOL_ACCEPT * abs(F_row[j])
            si = slice(i * g, (i + 1) * g)
            qg, qo, qold = Qg[j, si], res.Q[j, si], Q[j, si]
            if not np.array_equal(qg, qold) and not np.array_equal(qo, qold):
                # both accepted different proposals: the first difference in
                # back-substitution order must be a rounding near-tie
                l = int(np.nonzero(qg != qo)[0].max())
                ok = bool(ties[l])
            else:
                ok = bool(ties.any()) or acc_tie
            if not ok:
                unexplained.append((int(j), i))
        records.append(dict(k=k, rows_differ=len(bad_rows), rel_S=rel_S,
                            unexplained=unexplained))
        assert not unexplained, f"iteration {k}: differences not at near-ties: {unexplained[:5]}"
        S, Q = res.S, res.Q
    return records
