// Bounded Babai proposal and acceptance for group i of every active row
// (Sec. 3.3.2, Eqs. conditional_residual, group_bils, group_qr,
// babai_update; App. E "Small scales").
//
// One warp per output row; lane t owns coordinates l = lane + 32 u.  The
// group factors L_i = R_i^T and R_i^{-1} are staged in shared memory.
//
// The recursion is evaluated relative to the row's current codes q:
// with (H r)_i from the phase product and y = R_i^{-T} (H r)_i / s,
//     v = R_i^{-T} [(H r)_i + s H_ii c] / s = y + R_i c,   c = q - z,
// so the pre-round value of Eq. babai_update is
//     z + x_l = q_l + (y_l - sum_{h>l} R_lh Delta_h) / R_ll,
// Delta_h = q^cand_h - q_h.  The running vector u = y - R Delta is updated
// only where Delta_l != 0.  The change of the group objective (Eq.
// group_bils) is dF = s^2 (||R Delta - y||^2 - ||y||^2)
// = s^2 sum_l (a_l - y_l)(a_l + y_l) with a_l = R_ll Delta_l - u_l, which
// is exactly zero when the proposal equals the current codes.  A proposal
// is kept iff it changes a code, dF is finite and dF < 0.
#include "jarq_internal.cuh"

namespace jarq {
namespace {

struct BabaiArgs {
    const float *hr;      // [kSplitK][p][g]
    const float *Lf, *Rinv;
    const float *W, *S;
    uint8_t *Q;
    const int32_t *Z;
    float *r;
    const int *active;
    double *dF_sweep;
    int *accepted;
    int p, d, g, i, qmax;
    float eps;
};

template <int NTL>
__global__ void __launch_bounds__(256) babai_kernel(BabaiArgs a) {
    extern __shared__ float smem[];
    const int g = a.g, G = a.d / a.g;
    float *Lg = smem;           // [g][g] lower factor of group i
    float *Rg = smem + g * g;   // [g][g] R_i^{-1}
    const float *Lsrc = a.Lf + (size_t)a.i * g * g;
    const float *Rsrc = a.Rinv + (size_t)a.i * g * g;
    for (int idx = threadIdx.x; idx < g * g; idx += blockDim.x) {
        Lg[idx] = Lsrc[idx];
        Rg[idx] = Rsrc[idx];
    }
    __syncthreads();
    const int lane = threadIdx.x & 31, wpb = blockDim.x >> 5;
    const int col0 = a.i * g;
    for (int j = blockIdx.x * wpb + (threadIdx.x >> 5); j < a.p; j += gridDim.x * wpb) {
        if (!a.active[j]) continue;
        const float s = a.S[(size_t)j * G + a.i];
        if (!(fabsf(s) > a.eps)) continue;  // small-scale skip (also NaN)
        const int z = a.Z[(size_t)j * G + a.i];
        const size_t off = (size_t)j * a.d + col0;
        float hv[NTL], y[NTL], u[NTL];
        int qc[NTL], qn[NTL];
#pragma unroll
        for (int t = 0; t < NTL; ++t) {
            const int l = lane + 32 * t;
            float acc = 0.f;
            int q = 0;
            if (l < g) {
#pragma unroll
                for (int sp = 0; sp < kSplitK; ++sp)
                    acc += a.hr[((size_t)sp * a.p + j) * g + l];
                q = a.Q[off + l];
            }
            hv[t] = acc;
            qc[t] = q;
            qn[t] = q;
            y[t] = 0.f;
        }
        // y = R^{-T} (H r)_i / s :  y_l = sum_{m <= l} Rinv[m][l] hr_m
#pragma unroll
        for (int tt = 0; tt < NTL; ++tt) {
            for (int ml = 0; ml < 32; ++ml) {
                const int m = 32 * tt + ml;
                if (m >= g) break;
                const float hm = __shfl_sync(0xffffffffu, hv[tt], ml);
#pragma unroll
                for (int t = 0; t < NTL; ++t) {
                    const int l = lane + 32 * t;
                    if (t >= tt && l < g) y[t] = fmaf(Rg[m * g + l], hm, y[t]);
                }
            }
        }
#pragma unroll
        for (int t = 0; t < NTL; ++t) {
            y[t] = y[t] / s;
            u[t] = y[t];
        }
        // back substitution l = g-1 .. 0 (Eq. babai_update)
        int any = 0;
#pragma unroll
        for (int tt = NTL - 1; tt >= 0; --tt) {
            for (int ll = 31; ll >= 0; --ll) {
                const int l = 32 * tt + ll;
                if (l >= g) continue;
                int dl = 0;
                if (lane == ll) {
                    const float x = (float)qc[tt] + u[tt] / Lg[l * g + l];
                    float q = rintf(x);
                    q = fminf(fmaxf(q, 0.f), (float)a.qmax);
                    qn[tt] = (int)q;
                    dl = qn[tt] - qc[tt];
                }
                dl = __shfl_sync(0xffffffffu, dl, ll);
                if (dl != 0) {
                    any = 1;
                    const float fd = (float)dl;
#pragma unroll
                    for (int t = 0; t <= tt; ++t) {
                        const int lp = lane + 32 * t;
                        if (lp < l) u[t] = fmaf(-Lg[l * g + lp], fd, u[t]);
                    }
                }
            }
        }
        if (!any) continue;
        float acc = 0.f;
#pragma unroll
        for (int t = 0; t < NTL; ++t) {
            const int l = lane + 32 * t;
            if (l < g) {
                const float av = Lg[l * g + l] * (float)(qn[t] - qc[t]) - u[t];
                acc = fmaf(av - y[t], av + y[t], acc);
            }
        }
        for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        const float dF = s * s * acc;
        if (!(isfinite(dF) && dF < 0.f)) continue;
#pragma unroll
        for (int t = 0; t < NTL; ++t) {
            const int l = lane + 32 * t;
            if (l < g && qn[t] != qc[t]) {
                a.Q[off + l] = (uint8_t)qn[t];
                a.r[off + l] = fmaf(-s, (float)(qn[t] - z), a.W[off + l]);
            }
        }
        if (lane == 0) {
            a.dF_sweep[j] += (double)dF;
            a.accepted[j] += 1;
        }
    }
}

}  // namespace

cudaError_t launch_babai(const float *hr, const float *Lf, const float *Rinv, const float *W,
                         const float *S, uint8_t *Q, const int32_t *Z, float *r,
                         const int *active, double *dF_sweep, int *accepted, int p, int d,
                         int g, int i, int qmax, float eps, cudaStream_t s) {
    BabaiArgs a{hr, Lf, Rinv, W, S, Q, Z, r, active, dF_sweep, accepted, p, d, g, i, qmax, eps};
    const size_t smem = (size_t)2 * g * g * sizeof(float);
    const int wpb = 8;
    int blocks = (p + wpb - 1) / wpb;
    const int cap = num_sms() * (smem > 100 * 1024 ? 1 : 2);
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    cudaError_t e = cudaSuccess;
    const int ntl = (g + 31) / 32;
#define JARQ_BABAI_CASE(N)                                                                   \
    case N:                                                                                  \
        e = cudaFuncSetAttribute(babai_kernel<N>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                 (int)smem);                                                 \
        if (e != cudaSuccess) return e;                                                      \
        babai_kernel<N><<<blocks, 32 * wpb, smem, s>>>(a);                                   \
        break;
    switch (ntl) {
        JARQ_BABAI_CASE(1)
        JARQ_BABAI_CASE(2)
        JARQ_BABAI_CASE(3)
        JARQ_BABAI_CASE(4)
        default:
            return cudaErrorInvalidValue;
    }
#undef JARQ_BABAI_CASE
    return cudaGetLastError();
}

}  // namespace jarq
