// Bounded Babai proposal and acceptance for group i of output rows (Sec.
// 3.3.2, Eqs. conditional_residual, group_bils, group_qr, babai_update; App.
// E "Small scales"), executed by one warp.
//
// Lane l owns the NT = g/32 consecutive coordinates NT*l .. NT*l + NT - 1.
// The group factor L_i = R_i^T (row-major g x g, float32) is in shared
// memory.
//
// The recursion is evaluated relative to the row's current codes q.  The
// target y = R_i^{-T} (H r)_i / s is formed in double-float as
// (Pt_i - T_i) / s: Pt_i = R_i^{-T} (H w)_i from the folded target projection
// and T_i = sum_h s_h R_i^{-T} H_ih c_h from the phase product (split-K
// partials), so that the cancellation of H's low-rank part costs no
// precision.  Then
//     v = R_i^{-T} [(H r)_i + s H_ii c] / s = y + R_i c,   c = q - z,
// so the pre-round value of Eq. babai_update is
//     z + x_l = q_l + (y_l - sum_{h>l} R_lh Delta_h) / R_ll,
// Delta_h = q^cand_h - q_h.  The running vector u = y - R Delta changes only
// where Delta != 0.  The back substitution scans h = g-1 .. 0: the lane that
// owns coordinate h rounds it, the change is broadcast, and only when it is
// non-zero do the coordinates below take the column update (a warp-uniform
// branch).  A row none of whose codes would change at u = y has no change
// at all (the first coordinate's value is final and unchanged, and so on
// down) and skips the scan.
//
// The change of the group objective (Eq. group_bils) is
// dF = s^2 (||R Delta - y||^2 - ||y||^2) = s^2 sum_l (a_l - y_l)(a_l + y_l)
// with a_l = R_ll Delta_l - u_l, exactly zero for an unchanged proposal.  A
// proposal is kept iff it changes a code, dF is finite and dF < 0.
#pragma once

#include "jarq_internal.cuh"

namespace jarq {

struct BabaiRowArgs {
    const float *t_hi, *t_lo;    // [nsplit][p_pad][g] split-K partials of T_i
    const float *pt_hi, *pt_lo;  // [p][d] folded target projection Pt
    int nsplit;
    const float *S;              // [p][G]
    uint8_t *Q;                  // [p][d]
    const int32_t *Z;            // [p][G]
    __half *cplane;              // [p_pad][d_pad] codes c = q - z
    const int *active;
    int *accepted;
    int p_pad, d, d_pad, g, G, qmax;
    float eps;
};

template <int NT>
__device__ __forceinline__ void load_vec(const float *p, float (&v)[NT]) {
    if constexpr (NT == 4) {
        const float4 t = *reinterpret_cast<const float4 *>(p);
        v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
    } else if constexpr (NT == 2) {
        const float2 t = *reinterpret_cast<const float2 *>(p);
        v[0] = t.x; v[1] = t.y;
    } else {
#pragma unroll
        for (int k = 0; k < NT; ++k) v[k] = p[k];
    }
}

// The same through L2 only: the split-K partials may have been written by
// another thread block since this SM last cached them.
template <int NT>
__device__ __forceinline__ void load_vec_cg(const float *p, float (&v)[NT]) {
    if constexpr (NT == 4) {
        const float4 t = __ldcg(reinterpret_cast<const float4 *>(p));
        v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
    } else if constexpr (NT == 2) {
        const float2 t = __ldcg(reinterpret_cast<const float2 *>(p));
        v[0] = t.x; v[1] = t.y;
    } else {
#pragma unroll
        for (int k = 0; k < NT; ++k) v[k] = __ldcg(p + k);
    }
}

// Proposal and acceptance of group i for R rows at once (js[r] < 0: no
// row), their back substitutions interleaved so that one warp keeps R
// independent dependency chains in flight.
//
// The scan is blocked by lanes: for lane block L (coordinates h = NT L + t)
// the owning lane resolves its NT coordinates from the top one down, each
// rounding followed by the column updates of its own lower coordinates with
// the factor entries it holds in registers (Rl); then the NT changes are
// broadcast and the lanes below L apply the NT column updates, in the same
// descending order, from columns loaded before the broadcast.  Every u value
// sees the same fused multiply-adds in the same order as the
// coordinate-by-coordinate recursion (an update by a zero change leaves u
// unchanged), so the codes are those of Eq. babai_update evaluated in that
// order.
//   Lg: L_i in shared memory; rd: 1 / R_ll and dg: R_ll of this lane's
//   coordinates; Rl[t][tt] = R[l0+tt][l0+t] for tt < t (this lane's block
//   of the factor).
template <int NT, int R>
__device__ __forceinline__ void babai_rows(const BabaiRowArgs &a, const int (&js)[R], int i,
                                           const float *Lg, const float (&rd)[NT],
                                           const float (&dg)[NT], const float (&Rl)[NT][NT],
                                           int lane) {
    constexpr int g = 32 * NT;
    const int G = a.G, d = a.d;
    const int l0 = NT * lane;
    const int col0 = i * g;
    bool live[R];
    float s[R];
    int z[R];
    size_t off[R];
    float y[R][NT], u[R][NT], qc[R][NT], qn[R][NT];
#pragma unroll
    for (int r = 0; r < R; ++r) {
        const int j = js[r] >= 0 ? js[r] : 0;
        live[r] = js[r] >= 0 && a.active[j];
        s[r] = a.S[(size_t)j * G + i];
        live[r] = live[r] && fabsf(s[r]) > a.eps;   // small-scale skip (also NaN)
        z[r] = a.Z[(size_t)j * G + i];
        off[r] = (size_t)j * d + col0;
        // s y = Pt_i - sum_sp T_sp, in double-float
        float yl[NT];
        load_vec<NT>(a.pt_hi + off[r] + l0, y[r]);
        load_vec<NT>(a.pt_lo + off[r] + l0, yl);
        for (int sp = 0; sp < a.nsplit; ++sp) {
            float th[NT], tl[NT];
            const size_t o = ((size_t)sp * a.p_pad + j) * g + l0;
            load_vec_cg<NT>(a.t_hi + o, th);
            load_vec_cg<NT>(a.t_lo + o, tl);
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                const float sm = y[r][t] - th[t];
                const float bb = sm - y[r][t];
                const float e = (y[r][t] - (sm - bb)) + (-th[t] - bb);
                y[r][t] = sm;
                yl[t] += e - tl[t];
            }
        }
        uint32_t packed = 0;
        if constexpr (NT == 4) {
            packed = *reinterpret_cast<const uint32_t *>(a.Q + off[r] + l0);
        } else {
            packed = *reinterpret_cast<const uint16_t *>(a.Q + off[r] + l0);
        }
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            y[r][t] += yl[t];
            qc[r][t] = (float)((packed >> (8 * t)) & 0xFFu);   // small integers, exact
            qn[r][t] = qc[r][t];
        }
    }
    // y = R^{-T} (H r)_i / s; u = y
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            y[r][t] = y[r][t] / s[r];
            u[r][t] = y[r][t];
        }
    // back substitution (Eq. babai_update).  Rounding to the nearest even
    // integer adds and subtracts 1.5 * 2^23 (exact for |x| < 2^22; beyond
    // that the clamp to [0, qmax] gives the same code as rintf).
    const float qmaxf = (float)a.qmax;
    constexpr float kRound = 12582912.0f;      // 1.5 * 2^23
    bool scan[R], any[R];
    bool scan_any = false;
#pragma unroll
    for (int r = 0; r < R; ++r) {
        // does any code change at u = y?  If not, none changes at all.
        int nchg = 0;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            const float x = fmaf(u[r][t], rd[t], qc[r][t]);
            const float q = __fsub_rn(__fadd_rn(x, kRound), kRound);
            nchg += fminf(fmaxf(q, 0.f), qmaxf) != qc[r][t];
        }
        scan[r] = __any_sync(0xffffffffu, live[r] && nchg != 0);
        any[r] = false;
        scan_any |= scan[r];
    }
    if (scan_any) {
#pragma unroll 1
        for (int L = 31; L >= 0; --L) {
            // columns h = NT L + t of R for this lane's coordinates, loaded
            // before the changes are known (lanes below L only)
            float col[NT][NT];
            if (lane < L) {
#pragma unroll
                for (int t = 0; t < NT; ++t) load_vec<NT>(Lg + (NT * L + t) * g + l0, col[t]);
            }
            float dq[R][NT];
#pragma unroll
            for (int r = 0; r < R; ++r)
#pragma unroll
                for (int t = 0; t < NT; ++t) dq[r][t] = 0.f;
            if (lane == L) {
#pragma unroll
                for (int r = 0; r < R; ++r) {
                    if (!scan[r]) continue;
#pragma unroll
                    for (int t = NT - 1; t >= 0; --t) {
                        const float x = fmaf(u[r][t], rd[t], qc[r][t]);
                        const float q = fminf(fmaxf(__fsub_rn(__fadd_rn(x, kRound), kRound), 0.f),
                                              qmaxf);
                        dq[r][t] = q - qc[r][t];
                        qn[r][t] = q;
#pragma unroll
                        for (int tt = 0; tt < t; ++tt)
                            u[r][tt] = fmaf(-Rl[t][tt], dq[r][t], u[r][tt]);
                    }
                }
            }
#pragma unroll
            for (int r = 0; r < R; ++r)
#pragma unroll
                for (int t = 0; t < NT; ++t) dq[r][t] = __shfl_sync(0xffffffffu, dq[r][t], L);
#pragma unroll
            for (int r = 0; r < R; ++r) {
                bool nz = false;
#pragma unroll
                for (int t = 0; t < NT; ++t) nz |= dq[r][t] != 0.f;
                if (nz) {                                   // warp-uniform
                    any[r] = true;
                    if (lane < L) {
#pragma unroll
                        for (int t = NT - 1; t >= 0; --t)
#pragma unroll
                            for (int tt = 0; tt < NT; ++tt)
                                u[r][tt] = fmaf(-col[t][tt], dq[r][t], u[r][tt]);
                    }
                }
            }
        }
    }
    // dF = s^2 (||R Delta - y||^2 - ||y||^2) (Eq. group_bils); keep iff < 0
#pragma unroll
    for (int r = 0; r < R; ++r) {
        if (!any[r]) continue;                              // warp-uniform
        float acc = 0.f;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            const float av = dg[t] * (qn[r][t] - qc[r][t]) - u[r][t];
            acc = fmaf(av - y[r][t], av + y[r][t], acc);
        }
        for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        const float dF = s[r] * s[r] * acc;
        if (!(isfinite(dF) && dF < 0.f)) continue;
        const int j = js[r];
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            if (qn[r][t] != qc[r][t]) {
                const int l = l0 + t;
                const int qi = (int)qn[r][t];
                a.Q[off[r] + l] = (uint8_t)qi;
                a.cplane[(size_t)j * a.d_pad + col0 + l] = __int2half_rn(qi - z[r]);
            }
        }
        if (lane == 0) a.accepted[j] += 1;
    }
}

// This lane's part of the group factor for babai_rows: 1 / R_ll, R_ll and
// the lane's diagonal block.
template <int NT>
__device__ __forceinline__ void babai_lane_factor(const float *Lg, int lane, float (&rd)[NT],
                                                  float (&dg)[NT], float (&Rl)[NT][NT]) {
    constexpr int g = 32 * NT;
    const int l0 = NT * lane;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        dg[t] = Lg[(l0 + t) * g + l0 + t];
        rd[t] = 1.0f / dg[t];
#pragma unroll
        for (int tt = 0; tt < NT; ++tt) Rl[t][tt] = tt < t ? Lg[(l0 + t) * g + l0 + tt] : 0.f;
    }
}

}  // namespace jarq
