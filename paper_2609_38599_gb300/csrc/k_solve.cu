// Joint scale solve, one warp per output row (Sec. 3.3.1; App. E).
//
// For each active row j the warp
//  1. reads its G x G Gram matrix -- symmetric by construction, since the
//     Gram kernel computes each block once and writes it to both triangles,
//     so the symmetrisation of App. E "Solving for scales" is the identity
//     on it -- and forms, in float64, the gradient g = rhs - Gram s_old of
//     the current scales (rhs_i = c_i^T P_i from the target projection) and
//     the objective F(s_old) = wHw - s_old^T (rhs + g);
//  2. factors the Gram matrix by Cholesky in float32 (the paper solves this
//     system in FP32).  A pivot at or below rcond * max(max diag, eps), a
//     nonfinite entry or a failed factorisation adds ridge * I and retries
//     once; a second failure marks the row numerical and keeps its state;
//  3. solves the normal equations of Eq. scale_normal_equations for the
//     increment of the scales: Gram s_new = rhs <=> Gram (s_new - s_old) = g,
//     and with the ridge (Gram + lambda I) delta = g - lambda s_old (float32
//     Cholesky, then two refinement steps whose residuals are formed in
//     float64), and stores s_new rounded to float32;
//  4. evaluates L^{(k)} = F(s_new) = wHw - 2 s_new^T rhs + s_new^T Gram s_new
//     at the stored float32 scales and applies the early stop of Eq.
//     strict_stopping against L^{(k-1)}; with the ridge-acceptance option a
//     ridge-stabilised s_new that would raise F is dropped (App. G Remark
//     ridge-acceptance).
// In evaluation mode it only writes F(s) of the current state, for every
// row.
#include <float.h>

#include "jarq_internal.cuh"

namespace jarq {
namespace {

// In-place lower Cholesky of a G x G matrix (row stride G+1) by one warp.
// Fails when a pivot is not above `thr` or is not finite.  Each lane owns
// the rows a = lane (mod 32) of the trailing update; A[b][k] is read by all
// lanes at once (a broadcast) and the rows a differ in bank (stride G + 1).
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
        for (int a = k + 1 + lane; a < G; a += 32) {
            const float lak = A[a * ld + k];
            for (int b = k + 1; b <= a; ++b) A[a * ld + b] = fmaf(-lak, A[b * ld + k], A[a * ld + b]);
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
    const double *gram, *rhs, *wHw;
    float *S;
    double *L_prev;
    double *L_out;       // optional: F(s_old) of every processed row
    int *active, *iters, *ridge, *rstat, *status;
    int p, d, g, k;
    bool eval_only;
    jarq_options o;
};

// Per-warp shared memory: float A[G][G+1], s_old[G], work[G]; double g[G], inc[G].
__host__ __device__ inline size_t solve_warp_bytes(int G) {
    size_t f = (size_t)G * (G + 1) + 2 * (size_t)G;
    f = (f + 1) & ~(size_t)1;   // 8-byte alignment of the double part
    return f * sizeof(float) + 2 * (size_t)G * sizeof(double);
}

// Forward and back substitution with the float32 factor in A: y <- (L L^T)^{-1} y.
__device__ void warp_chol_solve(const float *A, int G, float *y) {
    const int lane = threadIdx.x & 31, ld = G + 1;
    for (int k = 0; k < G; ++k) {
        __syncwarp();
        const float yk = y[k] / A[k * ld + k];
        __syncwarp();
        if (lane == 0) y[k] = yk;
        for (int t = k + 1 + lane; t < G; t += 32) y[t] = fmaf(-A[t * ld + k], yk, y[t]);
    }
    for (int k = G - 1; k >= 0; --k) {
        __syncwarp();
        const float sk = y[k] / A[k * ld + k];
        __syncwarp();
        if (lane == 0) y[k] = sk;
        for (int t = lane; t < k; t += 32) y[t] = fmaf(-A[k * ld + t], sk, y[t]);
    }
    __syncwarp();
}

__global__ void scale_solve_kernel(SolveArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int G = a.d / a.g, ld = G + 1;
    const int wpb = blockDim.x >> 5, w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * wpb + w;
    if (j >= a.p || (!a.eval_only && !a.active[j])) return;  // warp-uniform
    unsigned char *base = smem_raw + (size_t)w * solve_warp_bytes(G);
    float *A = (float *)base;
    float *so = A + G * ld;         // s_old
    float *y = so + G;              // float work vector
    size_t fcount = (size_t)G * ld + 2 * (size_t)G;
    fcount = (fcount + 1) & ~(size_t)1;
    double *b = (double *)(base + fcount * sizeof(float));   // gradient g
    double *inc = b + G;                                      // increment of the scales
    const double *gj = a.gram + (size_t)j * G * G;
    const double *rj = a.rhs + (size_t)j * G;
    // the Gram matrix is exactly symmetric: entry (r0, c0) is read as
    // (c0, r0), so that lanes with consecutive r0 read consecutive addresses
    auto gsym = [&](int r0, int c0) { return gj[c0 * G + r0]; };
    for (int t = lane; t < G; t += 32) so[t] = a.S[(size_t)j * G + t];
    __syncwarp();
    // gradient g = rhs - Gram s_old and F(s_old) = wHw - s_old^T (rhs + g)
    bool bfin = true;
    double fs = 0.0;
    for (int r0 = lane; r0 < G; r0 += 32) {
        double gs = 0.0;
        for (int c0 = 0; c0 < G; ++c0) gs = fma(gsym(r0, c0), (double)so[c0], gs);
        const double gr = rj[r0] - gs;
        b[r0] = gr;
        fs += (double)so[r0] * (rj[r0] + gr);
        bfin &= (bool)isfinite(gr);
    }
    const double F_old = a.wHw[j] - warp_sum(fs);
    if (a.L_out && lane == 0) a.L_out[j] = F_old;
    if (a.eval_only) return;
    if (a.o.fixed_grid) {
        // fixed grid: the scales stay; L^(k) is the objective of the current state
        bool stop = false;
        if (a.o.early_stop && a.k >= 2) {
            const double dec = a.L_prev[j] - F_old;
            const double den = fmax(fabs(a.L_prev[j]), (double)a.o.eps);
            stop = (dec / den <= (double)a.o.tau_rel) || (fabs(dec) <= (double)a.o.tau_abs);
        }
        if (lane == 0) {
            a.L_prev[j] = F_old;
            a.iters[j] = a.k;
            if (stop) a.active[j] = 0;
        }
        return;
    }
    auto load_sym = [&](float shift) -> bool {
        bool finite = true;
        for (int r0 = 0; r0 < G; ++r0)
            for (int c0 = lane; c0 < G; c0 += 32) {
                float v = (float)gj[r0 * G + c0];
                if (r0 == c0) v += shift;
                if (!isfinite(v)) finite = false;
                A[r0 * ld + c0] = v;
            }
        __syncwarp();
        return __all_sync(0xffffffffu, finite);
    };
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
    ok = ok && __all_sync(0xffffffffu, bfin);
    auto fail = [&]() {
        if (lane == 0) {
            a.ridge[j] += used_ridge;
            a.rstat[j] = JARQ_ERR_NUMERICAL;
            a.active[j] = 0;
            atomicOr(a.status, ST_NUMERICAL);
        }
    };
    if (!ok) {
        fail();
        return;
    }
    // (Gram + lambda I) inc = g - lambda s_old, refined twice with float64 residuals
    const double lam = used_ridge ? (double)a.o.ridge : 0.0;
    for (int t = lane; t < G; t += 32) {
        inc[t] = 0.0;
        y[t] = (float)(b[t] - lam * (double)so[t]);
    }
    for (int step = 0; step < 3; ++step) {
        warp_chol_solve(A, G, y);
        for (int t = lane; t < G; t += 32) inc[t] += (double)y[t];
        __syncwarp();
        if (step == 2) break;
        for (int r0 = lane; r0 < G; r0 += 32) {
            double res = b[r0] - lam * ((double)so[r0] + inc[r0]);
            for (int c0 = 0; c0 < G; ++c0) res = fma(-gsym(r0, c0), inc[c0], res);
            y[r0] = (float)res;
        }
        __syncwarp();
    }
    bool sfin = true;
    for (int t = lane; t < G; t += 32) sfin &= (bool)isfinite(inc[t]);
    if (!__all_sync(0xffffffffu, sfin)) {
        fail();
        return;
    }
    for (int t = lane; t < G; t += 32) y[t] = (float)((double)so[t] + inc[t]);   // s_new
    __syncwarp();
    // L^{(k)} at the stored float32 scales, from the unridged symmetrised Gram
    double t1 = 0.0, t2 = 0.0;
    for (int r0 = lane; r0 < G; r0 += 32) {
        double gs = 0.0;
        for (int c0 = 0; c0 < G; ++c0) gs = fma(gsym(r0, c0), (double)y[c0], gs);
        t1 += (double)y[r0] * rj[r0];
        t2 += (double)y[r0] * gs;
    }
    double L_new = a.wHw[j] - 2.0 * warp_sum(t1) + warp_sum(t2);
    // Remark ridge-acceptance (optional): a ridge-stabilised solve that would
    // raise F_j is dropped and the previous scales stay
    const bool keep_old = used_ridge && a.o.ridge_accept && !(L_new <= F_old);
    if (keep_old) L_new = F_old;
    bool stop = false;
    if (a.o.early_stop && a.k >= 2) {
        const double dec = a.L_prev[j] - L_new;
        const double den = fmax(fabs(a.L_prev[j]), (double)a.o.eps);
        stop = (dec / den <= (double)a.o.tau_rel) || (fabs(dec) <= (double)a.o.tau_abs);
    }
    if (!keep_old)
        for (int t = lane; t < G; t += 32) a.S[(size_t)j * G + t] = y[t];
    if (lane == 0) {
        a.L_prev[j] = L_new;
        a.iters[j] = a.k;
        a.ridge[j] += used_ridge;
        if (stop) a.active[j] = 0;
    }
}

}  // namespace

cudaError_t launch_scale_solve(const double *gram, const double *rhs, const double *wHw, float *S,
                               double *L_prev, double *L_out, int *active,
                               int *iters, int *ridge, int *rstat, int *status, int p, int d,
                               int g, int k, bool eval_only, const jarq_options &o,
                               cudaStream_t s) {
    const int G = d / g;
    const size_t per_warp = solve_warp_bytes(G);
    int wpb = (int)((96 * 1024) / per_warp);
    if (wpb > 8) wpb = 8;
    if (wpb < 1) wpb = 1;
    const size_t smem = per_warp * wpb;
    cudaError_t e = cudaFuncSetAttribute(scale_solve_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    SolveArgs a{gram, rhs, wHw, S, L_prev, L_out, active, iters, ridge, rstat,
                status, p, d, g, k, eval_only, o};
    scale_solve_kernel<<<(p + wpb - 1) / wpb, 32 * wpb, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace jarq
