// Bounded Babai proposal and acceptance for group i of one output row (Sec.
// 3.3.2, Eqs. conditional_residual, group_bils, group_qr, babai_update; App.
// E "Small scales"), executed by one warp.  Used by the per-phase Babai
// kernel and by the fused sweep kernel.
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

// Proposal and acceptance for row j, group i.  Lg: L_i in shared memory;
// rd: 1 / R_ll of this lane's coordinates.  Returns true when the row's codes
// of group i changed.
template <int NT>
__device__ __forceinline__ bool babai_row(const BabaiRowArgs &a, int j, int i, const float *Lg,
                                          const float (&rd)[NT], int lane) {
    constexpr int g = 32 * NT;
    const int G = a.G, d = a.d;
    const int l0 = NT * lane;
    const int col0 = i * g;
    if (!a.active[j]) return false;
    const float s = a.S[(size_t)j * G + i];
    if (!(fabsf(s) > a.eps)) return false;  // small-scale skip (also NaN)
    const int z = a.Z[(size_t)j * G + i];
    const size_t off = (size_t)j * d + col0;
    // s y = Pt_i - sum_sp T_sp, in double-float
    float y[NT], yl[NT];
    load_vec<NT>(a.pt_hi + off + l0, y);
    load_vec<NT>(a.pt_lo + off + l0, yl);
    for (int sp = 0; sp < a.nsplit; ++sp) {
        float th[NT], tl[NT];
        const size_t o = ((size_t)sp * a.p_pad + j) * g + l0;
        load_vec_cg<NT>(a.t_hi + o, th);
        load_vec_cg<NT>(a.t_lo + o, tl);
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            const float sm = y[t] - th[t];
            const float bb = sm - y[t];
            const float e = (y[t] - (sm - bb)) + (-th[t] - bb);
            y[t] = sm;
            yl[t] += e - tl[t];
        }
    }
#pragma unroll
    for (int t = 0; t < NT; ++t) y[t] += yl[t];
    float qc[NT], qn[NT];   // current and proposed codes (small integers, exact)
    {
        uint32_t packed = 0;
        if constexpr (NT == 4) {
            packed = *reinterpret_cast<const uint32_t *>(a.Q + off + l0);
        } else {
            packed = *reinterpret_cast<const uint16_t *>(a.Q + off + l0);
        }
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            qc[t] = (float)((packed >> (8 * t)) & 0xFFu);
            qn[t] = qc[t];
        }
    }
    // y = R^{-T} (H r)_i / s
    float u[NT];
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        y[t] = y[t] / s;
        u[t] = y[t];
    }
    // back substitution (Eq. babai_update).  Rounding to the nearest even
    // integer adds and subtracts 1.5 * 2^23 (exact for |x| < 2^22; beyond
    // that the clamp to [0, qmax] gives the same code as rintf).
    const float qmaxf = (float)a.qmax;
    constexpr float kRound = 12582912.0f;      // 1.5 * 2^23
    bool any = false;
    // does any code change at u = y?
    int nchg = 0;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        const float x = fmaf(u[t], rd[t], qc[t]);
        const float r = __fsub_rn(__fadd_rn(x, kRound), kRound);
        nchg += fminf(fmaxf(r, 0.f), qmaxf) != qc[t];
    }
    if (__any_sync(0xffffffffu, nchg != 0)) {
        // descending scan (Eq. babai_update), coordinate h = NT L + t
        for (int L = 31; L >= 0; --L) {
#pragma unroll
            for (int t = NT - 1; t >= 0; --t) {
                const int h = NT * L + t;
                float dq = 0.f;
                if (lane == L) {
                    const float x = fmaf(u[t], rd[t], qc[t]);
                    const float r = __fsub_rn(__fadd_rn(x, kRound), kRound);
                    const float q = fminf(fmaxf(r, 0.f), qmaxf);
                    dq = q - qc[t];
                    qn[t] = q;
                }
                dq = __shfl_sync(0xffffffffu, dq, L);
                if (dq != 0.f) {                      // warp-uniform
                    any = true;
                    float lr[NT];
                    load_vec<NT>(Lg + h * g + l0, lr);   // R[l'][h] for l' = l0..
#pragma unroll
                    for (int tt = 0; tt < NT; ++tt)
                        if (l0 + tt < h) u[tt] = fmaf(-lr[tt], dq, u[tt]);
                }
            }
        }
    }
    if (!any) return false;
    float acc = 0.f;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        const float av = Lg[(l0 + t) * g + l0 + t] * (qn[t] - qc[t]) - u[t];
        acc = fmaf(av - y[t], av + y[t], acc);
    }
    for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    const float dF = s * s * acc;
    if (!(isfinite(dF) && dF < 0.f)) return false;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        if (qn[t] != qc[t]) {
            const int l = l0 + t;
            const int qi = (int)qn[t];
            a.Q[off + l] = (uint8_t)qi;
            a.cplane[(size_t)j * a.d_pad + col0 + l] = __int2half_rn(qi - z);
        }
    }
    if (lane == 0) a.accepted[j] += 1;
    return true;
}

}  // namespace jarq
