// Bounded Babai proposal and acceptance for group i of every active row
// (Sec. 3.3.2, Eqs. conditional_residual, group_bils, group_qr,
// babai_update; App. E "Small scales").
//
// One warp per output row; lane owns the NT = g/32 consecutive coordinates
// l = NT*lane .. NT*lane + NT - 1.  The group factors L_i = R_i^T and
// R_i^{-1} are staged in shared memory.
//
// The recursion is evaluated relative to the row's current codes q:
// with (H r)_i from the phase product and y = R_i^{-T} (H r)_i / s,
//     v = R_i^{-T} [(H r)_i + s H_ii c] / s = y + R_i c,   c = q - z,
// so the pre-round value of Eq. babai_update is
//     z + x_l = q_l + (y_l - sum_{h>l} R_lh Delta_h) / R_ll,
// Delta_h = q^cand_h - q_h.  The running vector u = y - R Delta changes only
// where Delta != 0, so the back substitution proceeds by jumps: every still
// undecided coordinate rounds its current value in parallel, the highest one
// whose code changes is fixed, its column updates u below it, and the scan
// continues beneath it.  Every u_l receives exactly the updates, in the
// order, of the one-coordinate-at-a-time recursion; the number of serial
// steps is the number of changed codes plus one.
//
// The change of the group objective (Eq. group_bils) is
// dF = s^2 (||R Delta - y||^2 - ||y||^2) = s^2 sum_l (a_l - y_l)(a_l + y_l)
// with a_l = R_ll Delta_l - u_l, exactly zero for an unchanged proposal.  A
// proposal is kept iff it changes a code, dF is finite and dF < 0.
#include "jarq_internal.cuh"

namespace jarq {
namespace {

constexpr int kWarps = 16;

struct BabaiArgs {
    const float *hr;      // [nsplit][p_pad][g]
    int nsplit;
    const float *Lf, *Rinv;
    const float *W, *S;
    uint8_t *Q;
    const int32_t *Z;
    ResidualView rv;
    const int *active;
    double *dF_sweep;
    int *accepted;
    int p, g, i, qmax;
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

template <int NT>
__global__ void __launch_bounds__(32 * kWarps) babai_kernel(BabaiArgs a) {
    constexpr int g = 32 * NT;
    extern __shared__ __align__(16) float smem[];
    float *Lg = smem;                 // [g][g] lower factor of group i
    float *Rg = smem + g * g;         // [g][g] R_i^{-1}
    float *rdiag = Rg + g * g;        // [g] 1 / R_ll
    float *hbuf = rdiag + g;          // [kWarps][g] this warp's (H r)_i row
    const int d = a.rv.d, G = d / g;
    const float *Lsrc = a.Lf + (size_t)a.i * g * g;
    const float *Rsrc = a.Rinv + (size_t)a.i * g * g;
    for (int idx = threadIdx.x * 4; idx < g * g; idx += blockDim.x * 4) {
        *reinterpret_cast<float4 *>(Lg + idx) = *reinterpret_cast<const float4 *>(Lsrc + idx);
        *reinterpret_cast<float4 *>(Rg + idx) = *reinterpret_cast<const float4 *>(Rsrc + idx);
    }
    __syncthreads();
    for (int l = threadIdx.x; l < g; l += blockDim.x) rdiag[l] = 1.0f / Lg[l * g + l];
    __syncthreads();
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    float *hrow = hbuf + wid * g;
    const int l0 = NT * lane;
    const int col0 = a.i * g;
    float rd[NT];
    load_vec<NT>(rdiag + l0, rd);
    for (int j = blockIdx.x * kWarps + wid; j < a.p; j += gridDim.x * kWarps) {
        if (!a.active[j]) continue;
        const float s = a.S[(size_t)j * G + a.i];
        if (!(fabsf(s) > a.eps)) continue;  // small-scale skip (also NaN)
        const int z = a.Z[(size_t)j * G + a.i];
        const size_t off = (size_t)j * d + col0;
        float hv[NT];
        load_vec<NT>(a.hr + (size_t)j * g + l0, hv);
        for (int sp = 1; sp < a.nsplit; ++sp) {
            float t2[NT];
            load_vec<NT>(a.hr + ((size_t)sp * a.rv.p_pad + j) * g + l0, t2);
#pragma unroll
            for (int t = 0; t < NT; ++t) hv[t] += t2[t];
        }
        int qc[NT], qn[NT];
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            qc[t] = a.Q[off + l0 + t];
            qn[t] = qc[t];
        }
        __syncwarp();
#pragma unroll
        for (int t = 0; t < NT; ++t) hrow[l0 + t] = hv[t];
        __syncwarp();
        // y = R^{-T} (H r)_i / s :  y_l = sum_{m <= l} Rinv[m][l] hr_m
        float y[NT];
#pragma unroll
        for (int t = 0; t < NT; ++t) y[t] = 0.f;
        for (int m = 0; m < g; m += 4) {
            const float4 h4 = *reinterpret_cast<const float4 *>(hrow + m);
            const float hm[4] = {h4.x, h4.y, h4.z, h4.w};
#pragma unroll
            for (int mm = 0; mm < 4; ++mm) {
                float rr[NT];
                load_vec<NT>(Rg + (m + mm) * g + l0, rr);
#pragma unroll
                for (int t = 0; t < NT; ++t) y[t] = fmaf(rr[t], hm[mm], y[t]);
            }
        }
        float u[NT];
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            y[t] = y[t] / s;
            u[t] = y[t];
        }
        // back substitution by jumps (Eq. babai_update)
        int hi = g - 1;
        bool any = false;
        while (hi >= 0) {
            int dl[NT], best = -1;
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                const int l = l0 + t;
                dl[t] = 0;
                if (l <= hi) {
                    float q = rintf(fmaf(u[t], rd[t], (float)qc[t]));
                    q = fminf(fmaxf(q, 0.f), (float)a.qmax);
                    dl[t] = (int)q - qc[t];
                    if (dl[t] != 0) best = l;
                }
            }
            const int lstar = __reduce_max_sync(0xffffffffu, best);
            if (lstar < 0) break;
            const int owner = lstar / NT, ts = lstar - owner * NT;
            int mine = 0;
#pragma unroll
            for (int t = 0; t < NT; ++t)
                if (t == ts) mine = dl[t];
            const int dstar = __shfl_sync(0xffffffffu, mine, owner);
            if (lane == owner) {
#pragma unroll
                for (int t = 0; t < NT; ++t)
                    if (t == ts) qn[t] = qc[t] + dstar;
            }
            any = true;
            const float fd = (float)dstar;
            float lr[NT];
            load_vec<NT>(Lg + lstar * g + l0, lr);   // R[l'][l*] for l' = l0..
#pragma unroll
            for (int t = 0; t < NT; ++t)
                if (l0 + t < lstar) u[t] = fmaf(-lr[t], fd, u[t]);
            hi = lstar - 1;
        }
        if (!any) continue;
        float acc = 0.f;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            const float av = Lg[(l0 + t) * g + l0 + t] * (float)(qn[t] - qc[t]) - u[t];
            acc = fmaf(av - y[t], av + y[t], acc);
        }
        for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        const float dF = s * s * acc;
        if (!(isfinite(dF) && dF < 0.f)) continue;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            if (qn[t] != qc[t]) {
                const int l = l0 + t;
                a.Q[off + l] = (uint8_t)qn[t];
                store_residual(a.rv, j, col0 + l, fmaf(-s, (float)(qn[t] - z), a.W[off + l]));
                store_code(a.rv, j, col0 + l, qn[t] - z);
            }
        }
        if (lane == 0) {
            a.dF_sweep[j] += (double)dF;
            a.accepted[j] += 1;
        }
    }
}

}  // namespace

cudaError_t launch_babai(const float *hr, int nsplit, const float *Lf, const float *Rinv,
                         const float *W, const float *S, uint8_t *Q, const int32_t *Z,
                         ResidualView rv, const int *active, double *dF_sweep, int *accepted,
                         int p, int g, int i, int qmax, float eps, cudaStream_t s) {
    BabaiArgs a{hr, nsplit, Lf, Rinv, W, S, Q, Z, rv, active, dF_sweep, accepted, p, g, i, qmax, eps};
    const size_t smem = ((size_t)2 * g * g + g + (size_t)kWarps * g) * sizeof(float);
    int blocks = (p + kWarps - 1) / kWarps;
    const int cap = num_sms() * (smem > 110 * 1024 ? 1 : 2);
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    cudaError_t e = cudaSuccess;
    if (g == 128) {
        e = cudaFuncSetAttribute(babai_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        babai_kernel<4><<<blocks, 32 * kWarps, smem, s>>>(a);
    } else if (g == 64) {
        e = cudaFuncSetAttribute(babai_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        babai_kernel<2><<<blocks, 32 * kWarps, smem, s>>>(a);
    } else {
        return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace jarq
