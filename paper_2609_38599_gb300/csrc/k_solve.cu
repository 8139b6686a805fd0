// Joint scale solve, one warp per output row (Sec. 3.3.1; App. E).
//
// For each active row j the warp
//  1. symmetrises its G x G Gram matrix (App. E "Solving for scales");
//  2. factors it by Cholesky in float32 (the paper solves this system in
//     FP32).  A pivot at or below rcond * max(max diag, eps), a nonfinite
//     entry or a failed factorisation adds ridge * I and retries once; a
//     second failure marks the row numerical and keeps its state;
//  3. solves the normal equations of Eq. scale_normal_equations for the
//     increment of the scales: with rhs = B^T y and the gradient
//     g = rhs - Gram s_old, whose entries are g_i = c_i^T (H r)_i at the
//     current state, Gram s_new = rhs  <=>  Gram (s_new - s_old) = g.  With the
//     ridge, (Gram + lambda I) s_new = rhs  <=>  (Gram + lambda I) delta =
//     g - lambda s_old.  g comes from a direct product with the residual, so
//     the solve's rounding only touches the (small) increment;
//  4. updates the bookkeeping for the early stop of Eq. strict_stopping:
//     the objective change at fixed codes is
//     dF_scale = -2 delta^T g + delta^T Gram delta, L^{(k)} = F(s_old) + dF_scale,
//     and L^{(k-1)} - L^{(k)} = -(accepted Babai dF of sweep k-1) - dF_scale
//     is formed from small terms only;
//  5. rewrites the row's residual r = w - D_s (q - z) for the new scales.
#include <float.h>

#include "jarq_internal.cuh"

namespace jarq {
namespace {

// In-place lower Cholesky of a G x G matrix (row stride G+1) by one warp.
// Fails when a pivot is not above `thr` or is not finite.
__device__ bool warp_cholesky(float *A, int G, float thr) {
    const int lane = threadIdx.x & 31, ld = G + 1;
    for (int k = 0; k < G; ++k) {
        __syncwarp();
        const float piv = A[k * ld + k];
        if (!(piv > thr) || !isfinite(piv)) return false;
        const float lkk = sqrtf(piv);
        __syncwarp();
        if (lane == 0) A[k * ld + k] = lkk;
        for (int a = k + 1 + lane; a < G; a += 32) A[a * ld + k] /= lkk;
        __syncwarp();
        const int n = G - k - 1;
        for (int idx = lane; idx < n * n; idx += 32) {
            int a = k + 1 + idx / n, b = k + 1 + idx % n;
            if (b <= a) A[a * ld + b] = fmaf(-A[a * ld + k], A[b * ld + k], A[a * ld + b]);
        }
    }
    __syncwarp();
    return true;
}

__device__ __forceinline__ double warp_sum(double v) {
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float warp_max(float v) {
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

struct SolveArgs {
    const float *gram, *gvec, *W;
    const uint8_t *Q;
    const int32_t *Z;
    const double *F_start;
    float *S, *r;
    double *L_prev, *dF_sweep;
    int *active, *iters, *ridge, *rstat, *status;
    int p, d, g, k;
    jarq_options o;
};

__global__ void scale_solve_kernel(SolveArgs a) {
    extern __shared__ float smem[];
    const int G = a.d / a.g, ld = G + 1;
    const int wpb = blockDim.x >> 5, w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * wpb + w;
    if (j >= a.p || !a.active[j]) return;  // warp-uniform
    float *A = smem + (size_t)w * (G * ld + 4 * G);
    float *b = A + G * ld;       // gradient g
    float *so = b + G;           // s_old
    float *y = so + G;           // right-hand side, then the increment
    const float *gj = a.gram + (size_t)j * G * G;
    auto load_sym = [&](float shift) -> bool {
        bool finite = true;
        for (int idx = lane; idx < G * G; idx += 32) {
            int r0 = idx / G, c0 = idx % G;
            float v = 0.5f * (gj[r0 * G + c0] + gj[c0 * G + r0]);
            if (r0 == c0) v += shift;
            if (!isfinite(v)) finite = false;
            A[r0 * ld + c0] = v;
        }
        __syncwarp();
        return __all_sync(0xffffffffu, finite);
    };
    for (int t = lane; t < G; t += 32) {
        b[t] = a.gvec[(size_t)j * G + t];
        so[t] = a.S[(size_t)j * G + t];
    }
    bool finite = load_sym(0.f);
    float md = 0.f;
    for (int t = lane; t < G; t += 32) md = fmaxf(md, A[t * ld + t]);
    md = warp_max(md);
    bool ok = finite && warp_cholesky(A, G, a.o.rcond * fmaxf(md, a.o.eps));
    int used_ridge = 0;
    if (!ok) {
        used_ridge = 1;
        load_sym(a.o.ridge);
        ok = warp_cholesky(A, G, 0.f);
    }
    // b must be finite for a usable solve
    bool bfin = true;
    for (int t = lane; t < G; t += 32) bfin &= (bool)isfinite(b[t]);
    ok = ok && __all_sync(0xffffffffu, bfin);
    if (!ok) {
        if (lane == 0) {
            a.ridge[j] += used_ridge;
            a.rstat[j] = JARQ_ERR_NUMERICAL;
            a.active[j] = 0;
            atomicOr(a.status, ST_NUMERICAL);
        }
        return;
    }
    // forward: L y = g - lambda s_old
    const float lam = used_ridge ? a.o.ridge : 0.f;
    for (int t = lane; t < G; t += 32) y[t] = fmaf(-lam, so[t], b[t]);
    for (int k = 0; k < G; ++k) {
        __syncwarp();
        const float yk = y[k] / A[k * ld + k];
        __syncwarp();
        if (lane == 0) y[k] = yk;
        for (int t = k + 1 + lane; t < G; t += 32) y[t] = fmaf(-A[t * ld + k], yk, y[t]);
    }
    // backward: L^T s = y
    for (int k = G - 1; k >= 0; --k) {
        __syncwarp();
        const float sk = y[k] / A[k * ld + k];
        __syncwarp();
        if (lane == 0) y[k] = sk;
        for (int t = lane; t < k; t += 32) y[t] = fmaf(-A[k * ld + t], sk, y[t]);
    }
    __syncwarp();
    bool sfin = true;
    for (int t = lane; t < G; t += 32) sfin &= (bool)isfinite(y[t]);
    if (!__all_sync(0xffffffffu, sfin)) {
        if (lane == 0) {
            a.ridge[j] += used_ridge;
            a.rstat[j] = JARQ_ERR_NUMERICAL;
            a.active[j] = 0;
            atomicOr(a.status, ST_NUMERICAL);
        }
        return;
    }
    // objective bookkeeping with the unridged symmetrised Gram matrix
    double t1 = 0.0, t2 = 0.0;
    for (int r0 = lane; r0 < G; r0 += 32) {
        float gdl = 0.f;
        for (int c0 = 0; c0 < G; ++c0)
            gdl = fmaf(0.5f * (gj[r0 * G + c0] + gj[c0 * G + r0]), y[c0], gdl);
        t1 += (double)y[r0] * (double)b[r0];
        t2 += (double)y[r0] * (double)gdl;
    }
    t1 = warp_sum(t1);
    t2 = warp_sum(t2);
    const double dF_scale = -2.0 * t1 + t2;
    const double L_new = a.F_start[j] + dF_scale;
    bool stop = false;
    if (a.o.early_stop && a.k >= 2) {
        const double dec = -(a.dF_sweep[j] + dF_scale);
        const double den = fmax(fabs(a.L_prev[j]), (double)a.o.eps);
        stop = (dec / den <= (double)a.o.tau_rel) || (fabs(dec) <= (double)a.o.tau_abs);
    }
    __syncwarp();
    for (int t = lane; t < G; t += 32) y[t] = so[t] + y[t];   // s_new = s_old + delta
    __syncwarp();
    for (int t = lane; t < G; t += 32) a.S[(size_t)j * G + t] = y[t];
    if (lane == 0) {
        a.L_prev[j] = L_new;
        a.dF_sweep[j] = 0.0;
        a.iters[j] = a.k;
        a.ridge[j] += used_ridge;
        if (stop) a.active[j] = 0;
    }
    // residual for the new scales
    const size_t rowoff = (size_t)j * a.d;
    const int32_t *zj = a.Z + (size_t)j * G;
    for (int c0 = lane; c0 < a.d; c0 += 32) {
        const int grp = c0 / a.g;
        const float c = (float)((int)a.Q[rowoff + c0] - zj[grp]);
        a.r[rowoff + c0] = fmaf(-y[grp], c, a.W[rowoff + c0]);
    }
}

}  // namespace

cudaError_t launch_scale_solve(const float *gram, const float *gvec, const float *W,
                               const uint8_t *Q, const int32_t *Z, const double *F_start, float *S,
                               float *r, double *L_prev, double *dF_sweep, int *active,
                               int *iters, int *ridge, int *rstat, int *status, int p, int d,
                               int g, int k, const jarq_options &o, cudaStream_t s) {
    const int G = d / g;
    const size_t per_warp = (size_t)(G * (G + 1) + 4 * G) * sizeof(float);
    int wpb = (int)((96 * 1024) / per_warp);
    if (wpb > 8) wpb = 8;
    if (wpb < 1) wpb = 1;
    const size_t smem = per_warp * wpb;
    cudaError_t e = cudaFuncSetAttribute(scale_solve_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    SolveArgs a{gram, gvec, W, Q, Z, F_start, S, r, L_prev, dF_sweep, active, iters, ridge, rstat,
                status, p, d, g, k, o};
    scale_solve_kernel<<<(p + wpb - 1) / wpb, 32 * wpb, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace jarq
