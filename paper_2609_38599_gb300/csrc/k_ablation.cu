// Mechanism ablations of JARQ (App. "Refinement Mechanisms", Tab.
// mechanism-summary (a)): the scale fits that the joint fit is compared with,
// and the multi-code probe (single-code search, then one Babai proposal).
//
// Scale fits with the codes fixed, one warp per output row, float64:
//  * independent (Eq. independent-fit): s_i = c_i^T H_ii w_i / c_i^T H_ii c_i,
//    each group fitted to its own contribution; the numerators come from
//    own_rhs_kernel, the denominators are the Gram diagonal;
//  * coordinate descent: one scale at a time against the full residual,
//    s_i += c_i^T (H r)_i / c_i^T H_ii c_i with the gradient rhs - Gram s kept
//    current, groups in order, a given number of passes.
//  A group with c_i^T H_ii c_i = 0 keeps its scale.  The scales are stored
//  as float32 and the objective wHw - 2 s^T rhs + s^T Gram s is evaluated at
//  the stored values, before and after.
//
// Multi-code probe for one group i, one warp per row, float64 decisions:
//  (H r)_i = P_i - T_i from the exact target projection P = W H and the
//  exact tensor-core product T_i = sum_h s_h H_ih c_h; then single-code
//  updates (each coordinate in order moved to its best code when that
//  strictly lowers F, by dF = -2 D (H r)_l + D^2 H_ll with D = s (q' - q_l),
//  full passes until one moves nothing), then one bounded Babai proposal
//  from that state (Eq. babai_update with the float64 factor R_i = L_i^T),
//  kept iff its dF < 0.  The codes are not written back: the probe reports
//  the searched codes, the number of moves, the proposal's acceptance, the
//  number of codes it changes and its dF.
#include "jarq_internal.cuh"

namespace jarq {
namespace {

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

__device__ __forceinline__ double warp_sum(double v) {
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// own[j][i] = c_i^T H_ii w_i.  Grid (ceil(p / 32), G), 256 threads; H_ii in
// shared memory (row pitch g + 1); a warp handles four rows; lane owns
// coordinates k = lane + 32 m and forms (H_ii w_i)_k in double-float (each
// float32 product split exactly by an fma).
__global__ void own_rhs_kernel(const float *__restrict__ Hs, const float *__restrict__ W,
                               const uint8_t *__restrict__ Q, const int32_t *__restrict__ Z,
                               double *__restrict__ own, int p, int d, int g) {
    extern __shared__ float sH[];
    const int G = d / g, i = blockIdx.y, ld = g + 1;
    const int base = i * g;
    for (int idx = threadIdx.x; idx < g * g; idx += blockDim.x) {
        const int a = idx / g, b = idx % g;
        sH[a * ld + b] = Hs[(size_t)(base + a) * d + base + b];
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nk = g / 32;
    for (int r = 0; r < 4; ++r) {
        const int j = blockIdx.x * 32 + warp * 4 + r;
        if (j >= p) break;                                   // warp-uniform
        const float *w = W + (size_t)j * d + base;
        const float wl0 = w[lane], wl1 = nk > 1 ? w[lane + 32] : 0.f;
        const float wl2 = nk > 2 ? w[lane + 64] : 0.f, wl3 = nk > 3 ? w[lane + 96] : 0.f;
        double acc = 0.0;
        for (int m = 0; m < nk; ++m) {
            const int k = lane + 32 * m;
            float sh = 0.f, sl = 0.f;
            for (int l = 0; l < g; ++l) {
                const int src = l & 31, blk = l >> 5;
                const float wsel = blk == 0 ? wl0 : blk == 1 ? wl1 : blk == 2 ? wl2 : wl3;
                const float wl = __shfl_sync(0xffffffffu, wsel, src);
                const float h = sH[k * ld + l];
                const float pr = h * wl, pe = fmaf(h, wl, -pr);
                float s2, e2;
                two_sum(sh, pr, s2, e2);
                sh = s2;
                sl += e2 + pe;
            }
            const int c = (int)Q[(size_t)j * d + base + k] - Z[(size_t)j * G + i];
            acc += (double)c * ((double)sh + (double)sl);
        }
        acc = warp_sum(acc);
        if (lane == 0) own[(size_t)j * G + i] = acc;
    }
}

struct FitArgs {
    const float2 *gram;   // [p][G][G] float pairs (hi, lo)
    const double *rhs, *own, *wHw;
    float *S;
    double *F_before, *F_after;
    int p, G, method, passes;
};

// A row's Gram matrix read as float64: each entry is stored as a float
// pair (hi, lo), whose sum is exact in float64.
struct PairRow {
    const float2 *p;
    __device__ double operator[](size_t i) const {
        const float2 e = p[i];
        return (double)e.x + (double)e.y;
    }
};

// F(s) = wHw - 2 s^T rhs + s^T Gram s for the scales in s (shared memory).
__device__ double row_objective(PairRow gj, const double *rj, double wHw, const double *s,
                                int G) {
    const int lane = threadIdx.x & 31;
    double t = 0.0;
    for (int r = lane; r < G; r += 32) {
        double gs = 0.0;
        for (int c = 0; c < G; ++c) gs = fma(gj[r * G + c], s[c], gs);
        t += s[r] * (gs - 2.0 * rj[r]);
    }
    return wHw + warp_sum(t);
}

// One warp per row; per-warp shared memory: s [G], grad [G] (float64).
__global__ void scale_fit_kernel(FitArgs a) {
    extern __shared__ double sm[];
    const int wpb = blockDim.x >> 5, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * wpb + warp;
    if (j >= a.p) return;                                    // warp-uniform
    const int G = a.G;
    double *s = sm + (size_t)warp * 2 * G, *grad = s + G;
    const PairRow gj{a.gram + (size_t)j * G * G};
    const double *rj = a.rhs + (size_t)j * G;
    for (int t = lane; t < G; t += 32) s[t] = (double)a.S[(size_t)j * G + t];
    __syncwarp();
    const double Fb = row_objective(gj, rj, a.wHw[j], s, G);
    __syncwarp();
    if (a.method == JARQ_FIT_INDEPENDENT) {
        for (int t = lane; t < G; t += 32) {
            const double dd = gj[t * G + t];
            if (dd > 0.0) s[t] = a.own[(size_t)j * G + t] / dd;
        }
    } else {
        // gradient c_i^T (H r)_i = rhs - Gram s of the current scales
        for (int r = lane; r < G; r += 32) {
            double gs = 0.0;
            for (int c = 0; c < G; ++c) gs = fma(gj[r * G + c], s[c], gs);
            grad[r] = rj[r] - gs;
        }
        __syncwarp();
        for (int pass = 0; pass < a.passes; ++pass)
            for (int i = 0; i < G; ++i) {
                const double dd = gj[i * G + i];
                const double step = dd > 0.0 ? grad[i] / dd : 0.0;
                __syncwarp();
                for (int r = lane; r < G; r += 32) grad[r] -= gj[r * G + i] * step;
                if (lane == 0) s[i] += step;
                __syncwarp();
            }
    }
    __syncwarp();
    // store float32 scales; the objective at the stored values
    for (int t = lane; t < G; t += 32) {
        const float f = __double2float_rn(s[t]);
        a.S[(size_t)j * G + t] = f;
        s[t] = (double)f;
    }
    __syncwarp();
    const double Fa = row_objective(gj, rj, a.wHw[j], s, G);
    if (lane == 0) {
        a.F_before[j] = Fb;
        a.F_after[j] = Fa;
    }
}

struct ProbeArgs {
    const float *Phi, *Plo;      // [p][d] P = W H (double-float)
    const float *t_hi, *t_lo;    // [nsplit][p_pad][g] T_i = sum_h s_h H_ih c_h
    const float *Hs;             // [d][d]
    const double *L64;           // [G][g][g] lower factor L_i = R_i^T (float64)
    const float *S;
    const uint8_t *Q;
    const int32_t *Z;
    uint8_t *q_out;              // [p][g] codes after the single-code search
    int32_t *moves, *accepted, *changed;
    double *dF;
    int p, p_pad, d, g, i, nsplit, qmax;
    float eps;
};

constexpr int kProbeWarps = 8;

// Shared memory: H_ii (float32, pitch g + 1), L_i (float64, pitch g + 1),
// per warp v[g] and the proposal's codes [g] (float64).
__global__ void __launch_bounds__(32 * kProbeWarps) probe_kernel(ProbeArgs a) {
    extern __shared__ double psm[];
    const int g = a.g, ld = g + 1, G = a.d / g, base = a.i * g;
    double *sL = psm;                                        // [g][ld]
    float *sH = (float *)(sL + (size_t)g * ld);              // [g][ld]
    double *wbuf = (double *)(sH + (((size_t)g * ld + 1) & ~(size_t)1));
    for (int idx = threadIdx.x; idx < g * g; idx += blockDim.x) {
        const int r = idx / g, c = idx % g;
        sH[r * ld + c] = a.Hs[(size_t)(base + r) * a.d + base + c];
        sL[r * ld + c] = a.L64[(size_t)a.i * g * g + idx];
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nt = g / 32;
    double *v = wbuf + (size_t)warp * 2 * g, *qb = v + g;
    for (int j = blockIdx.x * kProbeWarps + warp; j < a.p; j += gridDim.x * kProbeWarps) {
        const double s = (double)a.S[(size_t)j * G + a.i];
        const double z = (double)a.Z[(size_t)j * G + a.i];
        double hr[4], q[4];
        for (int t = 0; t < nt; ++t) {
            const int l = lane + 32 * t;
            const size_t off = (size_t)j * a.d + base + l;
            double acc = (double)a.Phi[off] + (double)a.Plo[off];
            for (int sp = 0; sp < a.nsplit; ++sp) {
                const size_t o = ((size_t)sp * a.p_pad + j) * g + l;
                acc -= (double)a.t_hi[o] + (double)a.t_lo[o];
            }
            hr[t] = acc;
            q[t] = (double)a.Q[(size_t)j * a.d + base + l];
        }
        int moves = 0, acc_flag = 0, nchg = 0;
        double dF = 0.0;
        if (fabs(s) > (double)a.eps) {
            // ---- single-code search
            for (int guard = 0; guard < 64 * g; ++guard) {
                bool moved = false;
                for (int l = 0; l < g; ++l) {
                    const int owner = l & 31, t = l >> 5;
                    double best = 0.0, bq = 0.0;
                    if (lane == owner) {
                        const double ql = t == 0 ? q[0] : t == 1 ? q[1] : t == 2 ? q[2] : q[3];
                        const double hl = t == 0 ? hr[0] : t == 1 ? hr[1] : t == 2 ? hr[2] : hr[3];
                        const double Hll = (double)sH[l * ld + l];
                        bq = ql;
                        for (int c = 0; c <= a.qmax; ++c) {
                            const double D = s * ((double)c - ql);
                            const double f = -2.0 * D * hl + D * D * Hll;
                            if (f < best) {
                                best = f;
                                bq = (double)c;
                            }
                        }
                        bq -= ql;                            // code step
                    }
                    const double dq = __shfl_sync(0xffffffffu, bq, owner);
                    if (dq != 0.0) {
                        const double D = s * dq;
                        for (int tt = 0; tt < nt; ++tt)
                            hr[tt] -= D * (double)sH[(lane + 32 * tt) * ld + l];
                        if (lane == owner) {
                            if (t == 0) q[0] += dq; else if (t == 1) q[1] += dq;
                            else if (t == 2) q[2] += dq; else q[3] += dq;
                        }
                        moved = true;
                        ++moves;
                    }
                }
                if (!moved) break;
            }
            // ---- Babai proposal from the searched state:
            // A_i^T y = (H r)_i + s H_ii c, v = L_i^{-1} (A_i^T y) / s
            double tv[4];
            for (int t = 0; t < nt; ++t) {
                const int l = lane + 32 * t;
                double acc = hr[t];
                for (int m = 0; m < g; ++m) {
                    const int src = m & 31, tm = m >> 5;
                    const double qsel = tm == 0 ? q[0] : tm == 1 ? q[1] : tm == 2 ? q[2] : q[3];
                    const double cm = __shfl_sync(0xffffffffu, qsel, src) - z;
                    acc = fma(s * (double)sH[l * ld + m], cm, acc);
                }
                tv[t] = acc;
            }
            for (int t = 0; t < nt; ++t) v[lane + 32 * t] = tv[t];
            __syncwarp();
            // forward substitution L v = t, then v /= s
            for (int l = 0; l < g; ++l) {
                double part = 0.0;
                for (int m = lane; m < l; m += 32) part = fma(sL[l * ld + m], v[m], part);
                part = warp_sum(part);
                if (lane == 0) v[l] = (v[l] - part) / sL[l * ld + l];
                __syncwarp();
            }
            for (int t = 0; t < nt; ++t) v[lane + 32 * t] /= s;
            __syncwarp();
            // bounded nearest plane, l = g-1 .. 0, with R_lm = L_ml
            for (int l = g - 1; l >= 0; --l) {
                double part = 0.0;
                for (int m = l + 1 + lane; m < g; m += 32) part = fma(sL[m * ld + l], qb[m] - z, part);
                part = warp_sum(part);
                if (lane == 0) {
                    const double x = (v[l] - part) / sL[l * ld + l];
                    qb[l] = fmin(fmax(rint(z + x), 0.0), (double)a.qmax);
                }
                __syncwarp();
            }
            // dF = -2 D^T (H r)_i + D^T H_ii D, D = s (qb - q)
            double lin = 0.0, quad = 0.0;
            int chg = 0;
            for (int t = 0; t < nt; ++t) {
                const int l = lane + 32 * t;
                const double Dl = s * (qb[l] - q[t]);
                lin += Dl * hr[t];
                chg += qb[l] != q[t];
                double hd = 0.0;
                for (int m = 0; m < g; ++m) {
                    const int src = m & 31, tm = m >> 5;
                    const double qsel = tm == 0 ? q[0] : tm == 1 ? q[1] : tm == 2 ? q[2] : q[3];
                    const double qm = __shfl_sync(0xffffffffu, qsel, src);
                    hd = fma((double)sH[l * ld + m], s * (qb[m] - qm), hd);
                }
                quad += Dl * hd;
            }
            lin = warp_sum(lin);
            quad = warp_sum(quad);
            for (int o = 16; o; o >>= 1) chg += __shfl_xor_sync(0xffffffffu, chg, o);
            dF = -2.0 * lin + quad;
            acc_flag = (isfinite(dF) && dF < 0.0) ? 1 : 0;
            nchg = chg;
            __syncwarp();
        }
        for (int t = 0; t < nt; ++t)
            a.q_out[(size_t)j * g + lane + 32 * t] = (uint8_t)q[t];
        if (lane == 0) {
            a.moves[j] = moves;
            a.accepted[j] = acc_flag;
            a.changed[j] = nchg;
            a.dF[j] = dF;
        }
    }
}

}  // namespace

cudaError_t launch_own_rhs(const float *Hs, const float *W, const uint8_t *Q, const int32_t *Z,
                           double *own, int p, int d, int g, cudaStream_t s) {
    const size_t smem = (size_t)g * (g + 1) * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(own_rhs_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    own_rhs_kernel<<<dim3((p + 31) / 32, d / g), 256, smem, s>>>(Hs, W, Q, Z, own, p, d, g);
    return cudaGetLastError();
}

cudaError_t launch_scale_fit(const float2 *gram, const double *rhs, const double *own,
                             const double *wHw, float *S, double *F_before, double *F_after, int p,
                             int G, int method, int passes, cudaStream_t s) {
    const int wpb = 8;
    const size_t smem = (size_t)wpb * 2 * G * sizeof(double);
    FitArgs a{gram, rhs, own, wHw, S, F_before, F_after, p, G, method, passes};
    scale_fit_kernel<<<(p + wpb - 1) / wpb, 32 * wpb, smem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_probe(const float *Phi, const float *Plo, const float *t_hi, const float *t_lo,
                         const float *Hs, const double *L64, const float *S, const uint8_t *Q,
                         const int32_t *Z, uint8_t *q_out, int32_t *moves, int32_t *accepted,
                         int32_t *changed, double *dF, int p, int p_pad, int d, int g, int i,
                         int nsplit, int qmax, float eps, cudaStream_t s) {
    const size_t ld = (size_t)g + 1;
    const size_t fl = ((size_t)g * ld + 1) & ~(size_t)1;
    const size_t smem = (size_t)g * ld * sizeof(double) + fl * sizeof(float) +
                        (size_t)kProbeWarps * 2 * g * sizeof(double);
    cudaError_t e = cudaFuncSetAttribute(probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    ProbeArgs a{Phi, Plo, t_hi, t_lo, Hs, L64, S, Q, Z, q_out, moves, accepted, changed, dF,
                p, p_pad, d, g, i, nsplit, qmax, eps};
    int blocks = (p + kProbeWarps - 1) / kProbeWarps;
    if (blocks > 4 * num_sms()) blocks = 4 * num_sms();
    probe_kernel<<<blocks, 32 * kProbeWarps, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace jarq
