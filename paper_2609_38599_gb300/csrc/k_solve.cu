// Joint scale solve, one warp per output row (Sec. 3.3.1; App. E).
//
// For each active row j the warp
//  1. reads its G x G Gram matrix -- symmetric by construction, since the
//     Gram kernel computes each block once and writes it to both triangles,
//     so the symmetrisation of App. E "Solving for scales" is the identity
//     on it -- and forms, in double-float (the Gram entries arrive as
//     float pairs), the gradient g = rhs - Gram s_old of the current scales
//     (rhs_i = c_i^T P_i from the target projection) and the objective
//     F(s_old) = wHw - s_old^T (rhs + g);
//  2. factors the Gram matrix by Cholesky in float32 (the paper solves this
//     system in FP32).  A pivot at or below rcond * max(max diag, eps), a
//     nonfinite entry or a failed factorisation adds ridge * I and retries
//     once; a second failure marks the row numerical and keeps its state;
//  3. solves the normal equations of Eq. scale_normal_equations for the
//     increment of the scales: Gram s_new = rhs <=> Gram (s_new - s_old) = g,
//     and with the ridge (Gram + lambda I) delta = g - lambda s_old (float32
//     Cholesky, then two refinement steps whose residuals are formed in
//     double-float), and stores s_new rounded to float32;
//  4. evaluates L^{(k)} = F(s_new) = wHw - 2 s_new^T rhs + s_new^T Gram s_new
//     at the stored float32 scales and applies the early stop of Eq.
//     strict_stopping against L^{(k-1)}; with the ridge-acceptance option a
//     ridge-stabilised s_new that would raise F is dropped (App. G Remark
//     ridge-acceptance).
// In evaluation mode it only writes F(s) of the current state, for every
// row.
#include <float.h>

#include "df.cuh"
#include "jarq_internal.cuh"

namespace jarq {
namespace {

// Offset of row a of a lower triangle stored row by row (packed).
__device__ __forceinline__ int tri(int a) { return (a * (a + 1)) >> 1; }

// In-place lower Cholesky of a G x G matrix stored as a packed lower
// triangle, by one warp.  Fails when a pivot is not above `thr` or is not
// finite.  Each lane owns the rows a = lane (mod 32) of the trailing update;
// A[b][k] is read by all lanes at once (a broadcast).
__device__ bool warp_cholesky(float *A, int G, float thr) {
    const int lane = threadIdx.x & 31;
    for (int k = 0; k < G; ++k) {
        __syncwarp();
        const float piv = A[tri(k) + k];
        if (!(piv > thr) || !isfinite(piv)) return false;
        const float lkk = sqrtf(piv);
        __syncwarp();
        if (lane == 0) A[tri(k) + k] = lkk;
        for (int a = k + 1 + lane; a < G; a += 32) A[tri(a) + k] /= lkk;
        __syncwarp();
        for (int a = k + 1 + lane; a < G; a += 32) {
            float *Aa = A + tri(a);
            const float lak = Aa[k];
            // A[b][k] (rows b > k, column k) and A[a][b] (row a, columns
            // b > k) never overlap: four of each are loaded before the
            // four updates are stored
            int b = k + 1;
            for (; b + 3 <= a; b += 4) {
                const int t0 = tri(b) + k;
                const float c0 = A[t0], c1 = A[t0 + b + 1], c2 = A[t0 + 2 * b + 3],
                            c3 = A[t0 + 3 * b + 6];
                const float x0 = Aa[b], x1 = Aa[b + 1], x2 = Aa[b + 2], x3 = Aa[b + 3];
                Aa[b] = fmaf(-lak, c0, x0);
                Aa[b + 1] = fmaf(-lak, c1, x1);
                Aa[b + 2] = fmaf(-lak, c2, x2);
                Aa[b + 3] = fmaf(-lak, c3, x3);
            }
            for (; b <= a; ++b) Aa[b] = fmaf(-lak, A[tri(b) + k], Aa[b]);
        }
    }
    __syncwarp();
    return true;
}

__device__ __forceinline__ float warp_max(float v) {
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

struct SolveArgs {
    const float2 *gram;  // [p][G][G] Gram matrices as float pairs (hi, lo)
    const double *rhs, *wHw;
    float *S;
    double *L_prev;
    double *L_out;       // optional: F(s_old) of every processed row
    int *active, *iters, *ridge, *rstat, *status;
    int p, d, g, k;
    bool eval_only;
    jarq_options o;
};

// Per-warp shared memory: the packed lower factor A (G (G + 1) / 2
// floats), s_old[G], y[G], and the double-float gradient (bh, bl) and
// increment (ih, il), G each.
__host__ __device__ inline size_t solve_warp_bytes(int G) {
    return ((size_t)G * (G + 1) / 2 + 6 * (size_t)G) * sizeof(float);
}

// Forward and back substitution with the packed float32 factor in A,
// y <- (L L^T)^{-1} y, for G <= 128: lane l keeps y[l + 32 m] in a
// register, multiplies by the pivots' reciprocals, and each solved value
// reaches the other lanes by a shuffle.  y is read and written in shared
// memory.
__device__ void warp_chol_solve(const float *A, int G, float *y) {
    const int lane = threadIdx.x & 31;
    float v[4], rd[4];
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        const int t = lane + 32 * m;
        v[m] = t < G ? y[t] : 0.f;
        rd[m] = t < G ? 1.0f / A[tri(t) + t] : 0.f;
    }
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        for (int kk = 0; kk < 32; ++kk) {
            const int k = 32 * m + kk;
            if (k >= G) break;   // warp-uniform
            const float yk = __shfl_sync(0xffffffffu, v[m] * rd[m], kk);
            if (lane == kk) v[m] = yk;
#pragma unroll
            for (int mm = m; mm < 4; ++mm) {
                const int t = lane + 32 * mm;
                if (t > k && t < G) v[mm] = fmaf(-A[tri(t) + k], yk, v[mm]);
            }
        }
    }
#pragma unroll
    for (int m = 3; m >= 0; --m) {
        for (int kk = 31; kk >= 0; --kk) {
            const int k = 32 * m + kk;
            if (k >= G) continue;   // warp-uniform
            const float sk = __shfl_sync(0xffffffffu, v[m] * rd[m], kk);
            if (lane == kk) v[m] = sk;
#pragma unroll
            for (int mm = 0; mm <= m; ++mm) {
                const int t = lane + 32 * mm;
                if (t < k) v[mm] = fmaf(-A[tri(k) + t], sk, v[mm]);
            }
        }
    }
    __syncwarp();
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        const int t = lane + 32 * m;
        if (t < G) y[t] = v[m];
    }
    __syncwarp();
}

// Row r0 of the (exactly symmetric) Gram matrix times x = xh + xl, in
// double-float.  Entry (r0, c) is read as (c, r0), so that lanes with
// consecutive r0 read consecutive addresses, eight loads at a time.
template <bool kPair>
__device__ __forceinline__ DF gram_dot(const float2 *gj, int G, int r0, const float *xh,
                                       const float *xl) {
    DF acc{0.f, 0.f};
    auto term = [&](float2 e, int c) {
        df_add_prod(acc, e.x, xh[c]);
        acc.l = fmaf(e.y, xh[c], acc.l);
        if (kPair) acc.l = fmaf(e.x, xl[c], acc.l);
    };
    int c = 0;
    for (; c + 8 <= G; c += 8) {
        float2 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = __ldg(gj + (size_t)(c + u) * G + r0);
#pragma unroll
        for (int u = 0; u < 8; ++u) term(v[u], c + u);
    }
    for (; c < G; ++c) term(__ldg(gj + (size_t)c * G + r0), c);
    return acc;
}

// Solve for G > 32 (e.g. 86 groups of the 11008-input layers): the Gram
// matrix stays in global memory (L2) and is read row by row; the float32
// factor lives in shared memory.  Every dot product with the Gram matrix --
// the gradient, the two refinement residuals, the objective -- is summed in
// double-float on the entries' float pairs.
__global__ void scale_solve_kernel(SolveArgs a) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int G = a.d / a.g;
    const int wpb = blockDim.x >> 5, w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * wpb + w;
    if (j >= a.p || (!a.eval_only && !a.active[j])) return;  // warp-uniform
    float *A = (float *)(smem_raw + (size_t)w * solve_warp_bytes(G));
    float *so = A + tri(G);         // s_old
    float *y = so + G;              // float work vector
    float *bh = y + G, *bl = bh + G;    // gradient g (double-float)
    float *ih = bl + G, *il = ih + G;   // increment of the scales (double-float)
    const float2 *gj = a.gram + (size_t)j * G * G;
    const double *rj = a.rhs + (size_t)j * G;
    // the row's Gram matrix (8 G^2 bytes) is read by five or six passes:
    // bring it into L2 once, all lines at a time
    {
        const char *gb = (const char *)gj;
        const size_t bytes = (size_t)G * G * sizeof(double);
        for (size_t off = (size_t)lane * 128; off < bytes; off += 32 * 128)
            asm volatile("prefetch.global.L2 [%0];" ::"l"(gb + off));
        if (lane == 0) asm volatile("prefetch.global.L2 [%0];" ::"l"(gb + bytes - 1));
    }
    for (int t = lane; t < G; t += 32) so[t] = a.S[(size_t)j * G + t];
    __syncwarp();
    // gradient g = rhs - Gram s_old and F(s_old) = wHw - s_old^T (rhs + g)
    bool bfin = true;
    DF fs{0.f, 0.f};
    for (int r0 = lane; r0 < G; r0 += 32) {
        const DF gs = gram_dot<false>(gj, G, r0, so, nullptr);
        const DF rr = split_double(rj[r0]);
        const DF gr = df_add(rr, df_neg(gs));
        bh[r0] = gr.h;
        bl[r0] = gr.l;
        const DF rg = df_add(rr, gr);
        df_add_prod(fs, so[r0], rg.h);
        fs.l = fmaf(so[r0], rg.l, fs.l);
        bfin &= (bool)isfinite(gr.h);
    }
    const double F_old = a.wHw[j] - df_to_double(df_warp_sum(fs));
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
    // float32 copy of the Gram matrix (the high part of a pair is the
    // correctly rounded float32 of the entry), plus a ridge shift of the
    // diagonal
    auto load_sym = [&](float shift) -> bool {
        bool finite = true;
#pragma unroll 4
        for (int r0 = 0; r0 < G; ++r0)
            for (int c0 = lane; c0 <= r0; c0 += 32) {
                float v = __ldg(gj + (size_t)r0 * G + c0).x;
                if (r0 == c0) v += shift;
                if (!isfinite(v)) finite = false;
                A[tri(r0) + c0] = v;
            }
        __syncwarp();
        return __all_sync(0xffffffffu, finite);
    };
    bool finite = load_sym(0.f);
    float md = 0.f;
    for (int t = lane; t < G; t += 32) md = fmaxf(md, A[tri(t) + t]);
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
    // (Gram + lambda I) inc = g - lambda s_old, refined twice with
    // double-float residuals
    const float lam = used_ridge ? a.o.ridge : 0.f;
    for (int t = lane; t < G; t += 32) {
        ih[t] = 0.f;
        il[t] = 0.f;
        DF v{bh[t], bl[t]};
        df_add_prod(v, -lam, so[t]);
        y[t] = __fadd_rn(v.h, v.l);
    }
    for (int step = 0; step < 3; ++step) {
        warp_chol_solve(A, G, y);
        for (int t = lane; t < G; t += 32) {
            const DF s2 = df_add({ih[t], il[t]}, {y[t], 0.f});
            ih[t] = s2.h;
            il[t] = s2.l;
        }
        __syncwarp();
        if (step == 2) break;
        for (int r0 = lane; r0 < G; r0 += 32) {
            // res = g - lambda (s_old + inc) - Gram inc
            DF res{bh[r0], bl[r0]};
            df_add_prod(res, -lam, so[r0]);
            df_add_prod(res, -lam, ih[r0]);
            res.l = fmaf(-lam, il[r0], res.l);
            res = df_add(res, df_neg(gram_dot<true>(gj, G, r0, ih, il)));
            y[r0] = __fadd_rn(res.h, res.l);
        }
        __syncwarp();
    }
    bool sfin = true;
    for (int t = lane; t < G; t += 32) sfin &= (bool)(isfinite(ih[t]) && isfinite(il[t]));
    if (!__all_sync(0xffffffffu, sfin)) {
        fail();
        return;
    }
    // s_new = s_old + inc, rounded once to float32
    for (int t = lane; t < G; t += 32) {
        const DF s2 = df_add({so[t], 0.f}, {ih[t], il[t]});
        y[t] = __fadd_rn(s2.h, s2.l);
    }
    __syncwarp();
    // L^{(k)} at the stored float32 scales, from the unridged Gram matrix
    DF t1{0.f, 0.f}, t2{0.f, 0.f};
    for (int r0 = lane; r0 < G; r0 += 32) {
        const DF gs = gram_dot<false>(gj, G, r0, y, nullptr);
        const DF rr = split_double(rj[r0]);
        df_add_prod(t1, y[r0], rr.h);
        t1.l = fmaf(y[r0], rr.l, t1.l);
        df_add_prod(t2, y[r0], gs.h);
        t2.l = fmaf(y[r0], gs.l, t2.l);
    }
    double L_new = a.wHw[j] - 2.0 * df_to_double(df_warp_sum(t1)) + df_to_double(df_warp_sum(t2));
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


// ---------------------------------------------------------------------------
// Register-resident solve for G <= 32 (the g = 128 layers of 4096 inputs).
//
// Same steps, same decisions, no bulk float64: on GB300 float64 runs at
// about 1/64 of the float32 rate, so the dot products of the gradient, the
// refinement residuals and the objective are done in double-float (pairs of
// float32 with error-free products and sums, about 48 significant bits).
// Lane l owns row l of the Gram matrix (= column l: it is exactly
// symmetric) as the double-float pair per entry that the Gram kernel
// stores.  The float32 Cholesky keeps row l in registers and
// broadcasts the column of each step with shuffles: the same operations in
// the same order as warp_cholesky, so the factor (and the ridge decision)
// is bit-identical.  The triangular solves multiply by the reciprocal of
// the pivots; the float64-accurate refinement makes the stored scales
// independent of that rounding.
// ---------------------------------------------------------------------------

// In-place lower Cholesky with lane a holding row a in A[]; on and below
// the diagonal the operations and their order are those of warp_cholesky.
__device__ __forceinline__ bool reg_cholesky(float (&A)[32], int G, float thr) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int k = 0; k < 32; ++k) {
        if (k < G) {
            const float piv = __shfl_sync(0xffffffffu, A[k], k);
            if (!(piv > thr) || !isfinite(piv)) return false;   // warp-uniform
            const float lkk = sqrtf(piv);
            float lak = 0.f;
            if (lane > k) lak = A[k] / lkk;
            if (lane == k) A[k] = lkk;
            if (lane > k) A[k] = lak;
            // entries b <= a take the update of warp_cholesky; the entries
            // above the diagonal (b > a) are never read again, so they take
            // it as well instead of a predicate per entry
#pragma unroll
            for (int b = k + 1; b < 32; ++b) {
                const float lbk = __shfl_sync(0xffffffffu, lak, b);
                A[b] = fmaf(-lak, lbk, A[b]);
            }
        }
    }
    return true;
}

// y <- (L L^T)^{-1} y with lane a holding y_a; L row-major in Ls (stride
// 33) with zeros above the diagonal, dinv = 1 / L_aa.
__device__ __forceinline__ float reg_chol_solve(const float *Ls, int G, float dinv, float y) {
    const int lane = threadIdx.x & 31;
#pragma unroll 4
    for (int k = 0; k < G; ++k) {
        const float yk = __shfl_sync(0xffffffffu, __fmul_rn(y, dinv), k);
        const float t = fmaf(-Ls[lane * 33 + k], yk, y);   // lanes a < k: L_ak = 0
        y = lane == k ? yk : t;
    }
#pragma unroll 4
    for (int k = G - 1; k >= 0; --k) {
        const float xk = __shfl_sync(0xffffffffu, __fmul_rn(y, dinv), k);
        const float t = fmaf(-Ls[k * 33 + lane], xk, y);   // lanes a > k: L_ka = 0
        y = lane == k ? xk : t;
    }
    return y;
}

constexpr int kSmallWarps = 4;   // rows (warps) per block of the G <= 32 kernel

__global__ void __launch_bounds__(32 * kSmallWarps, 4) scale_solve_small_kernel(SolveArgs a) {
    __shared__ float Lsh[kSmallWarps][32 * 33];
    const int G = a.d / a.g;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kSmallWarps + w;
    if (j >= a.p) return;  // warp-uniform
    const bool own = lane < G;
    const float2 *gj = a.gram + (size_t)j * G * G;
    // row `lane` of the Gram matrix, read column-wise (coalesced) by
    // symmetry: every load (and the row's active flag) is issued before the
    // first is used
    const int act = a.eval_only ? 1 : a.active[j];
    DF gr[32];
#pragma unroll
    for (int c = 0; c < 32; ++c) {
        const float2 e = (own && c < G) ? gj[(size_t)c * G + lane] : make_float2(0.f, 0.f);
        gr[c] = DF{e.x, e.y};
    }
    const float so = own ? a.S[(size_t)j * G + lane] : 0.f;
    const double rhs_d = own ? a.rhs[(size_t)j * G + lane] : 0.0;
    if (!act) return;  // warp-uniform
    const DF rh = split_double(rhs_d);

    // gradient g = rhs - Gram s_old and F(s_old) = wHw - s_old^T (rhs + g)
    DF acc{0.f, 0.f};
#pragma unroll
    for (int c = 0; c < 32; ++c) {
        if (c < G) {
            const float sc = __shfl_sync(0xffffffffu, so, c);
            df_add_prod(acc, gr[c].h, sc);
            acc.l = __fmaf_rn(gr[c].l, sc, acc.l);
        }
    }
    const DF gd = df_add(rh, df_neg(acc));
    const bool bfin = isfinite(gd.h) && isfinite(gd.l);
    DF fs{0.f, 0.f};
    {
        const DF t = df_add(rh, gd);
        df_add_prod(fs, so, t.h);
        fs.l = __fmaf_rn(so, t.l, fs.l);
    }
    const double F_old = a.wHw[j] - df_to_double(df_warp_sum(fs));
    if (a.L_out && lane == 0) a.L_out[j] = F_old;
    if (a.eval_only) return;
    if (a.o.fixed_grid) {
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

    // float32 factor of the Gram matrix (entries rounded to nearest, as a
    // float64 -> float32 conversion does), with the ridge retry
    float A[32];
    bool finite = true;
    float diag = 0.f;
#pragma unroll
    for (int c = 0; c < 32; ++c) {
        A[c] = gr[c].h;
        finite &= (bool)isfinite(A[c]);
        if (c == lane) diag = A[c];
    }
    finite = __all_sync(0xffffffffu, finite);
    const float md = warp_max(own ? diag : 0.f);
    bool ok = finite && reg_cholesky(A, G, a.o.rcond * fmaxf(md, a.o.eps));
    int used_ridge = 0;
    if (!ok) {
        used_ridge = 1;
#pragma unroll
        for (int c = 0; c < 32; ++c) A[c] = (c == lane) ? gr[c].h + a.o.ridge : gr[c].h;
        ok = reg_cholesky(A, G, 0.f);
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
    float *Ls = Lsh[w];
    float ldiag = 1.f;
#pragma unroll
    for (int c = 0; c < 32; ++c) {
        Ls[lane * 33 + c] = c <= lane ? A[c] : 0.f;
        if (c == lane) ldiag = A[c];
    }
    __syncwarp();
    const float dinv = own ? 1.0f / ldiag : 0.f;

    // (Gram + lambda I) inc = g - lambda s_old, refined twice with
    // double-float residuals
    const float lam = used_ridge ? a.o.ridge : 0.f;
    DF b = gd;
    if (used_ridge) {
        df_add_prod(b, -lam, so);
    }
    DF inc{0.f, 0.f};
    float y = own ? __fadd_rn(b.h, b.l) : 0.f;
    for (int step = 0; step < 3; ++step) {
        y = reg_chol_solve(Ls, G, dinv, y);
        if (!own) y = 0.f;
        inc = df_add(inc, DF{y, 0.f});
        if (step == 2) break;
        DF res = b;
        if (used_ridge) {
            df_add_prod(res, -lam, inc.h);
            res.l = __fmaf_rn(-lam, inc.l, res.l);
        }
        DF q{0.f, 0.f};
#pragma unroll
        for (int c = 0; c < 32; ++c) {
            if (c < G) {
                const float ih = __shfl_sync(0xffffffffu, inc.h, c);
                const float il = __shfl_sync(0xffffffffu, inc.l, c);
                df_add_prod(q, gr[c].h, ih);
                q.l = __fmaf_rn(gr[c].h, il, q.l);
                q.l = __fmaf_rn(gr[c].l, ih, q.l);
            }
        }
        res = df_add(res, df_neg(q));
        y = own ? __fadd_rn(res.h, res.l) : 0.f;
    }
    if (!__all_sync(0xffffffffu, isfinite(inc.h) && isfinite(inc.l))) {
        fail();
        return;
    }
    // s_new = float32(s_old + inc)
    float sn = 0.f;
    if (own) {
        const DF t = df_two_sum(so, inc.h);
        sn = __fadd_rn(t.h, __fadd_rn(t.l, inc.l));
    }
    // L^{(k)} = wHw - 2 s^T rhs + s^T Gram s at the stored float32 scales
    DF gs{0.f, 0.f};
#pragma unroll
    for (int c = 0; c < 32; ++c) {
        if (c < G) {
            const float sc = __shfl_sync(0xffffffffu, sn, c);
            df_add_prod(gs, gr[c].h, sc);
            gs.l = __fmaf_rn(gr[c].l, sc, gs.l);
        }
    }
    DF t1{0.f, 0.f}, t2{0.f, 0.f};
    df_add_prod(t1, sn, rh.h);
    t1.l = __fmaf_rn(sn, rh.l, t1.l);
    df_add_prod(t2, sn, gs.h);
    t2.l = __fmaf_rn(sn, gs.l, t2.l);
    t1 = df_warp_sum(t1);
    t2 = df_warp_sum(t2);
    double L_new = a.wHw[j] - 2.0 * df_to_double(t1) + df_to_double(t2);
    const bool keep_old = used_ridge && a.o.ridge_accept && !(L_new <= F_old);
    if (keep_old) L_new = F_old;
    bool stop = false;
    if (a.o.early_stop && a.k >= 2) {
        const double dec = a.L_prev[j] - L_new;
        const double den = fmax(fabs(a.L_prev[j]), (double)a.o.eps);
        stop = (dec / den <= (double)a.o.tau_rel) || (fabs(dec) <= (double)a.o.tau_abs);
    }
    if (!keep_old && own) a.S[(size_t)j * G + lane] = sn;
    if (lane == 0) {
        a.L_prev[j] = L_new;
        a.iters[j] = a.k;
        a.ridge[j] += used_ridge;
        if (stop) a.active[j] = 0;
    }
}

}  // namespace

cudaError_t launch_scale_solve(const float2 *gram, const double *rhs, const double *wHw, float *S,
                               double *L_prev, double *L_out, int *active,
                               int *iters, int *ridge, int *rstat, int *status, int p, int d,
                               int g, int k, bool eval_only, const jarq_options &o,
                               cudaStream_t s) {
    const int G = d / g;
    SolveArgs a{gram, rhs, wHw, S, L_prev, L_out, active, iters, ridge, rstat,
                status, p, d, g, k, eval_only, o};
    if (G <= 32) {
        scale_solve_small_kernel<<<(p + kSmallWarps - 1) / kSmallWarps, 32 * kSmallWarps, 0, s>>>(a);
        return cudaGetLastError();
    }
    // at most four warps per block, and blocks small enough that several fit
    // on an SM: the kernel is bound by the latency of each warp's chain
    const size_t per_warp = solve_warp_bytes(G);
    int wpb = (int)((56 * 1024) / per_warp);
    if (wpb > 4) wpb = 4;
    if (wpb < 1) wpb = 1;
    const size_t smem = per_warp * wpb;
    cudaError_t e = cudaFuncSetAttribute(scale_solve_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    scale_solve_kernel<<<(p + wpb - 1) / wpb, 32 * wpb, smem, s>>>(a);
    return cudaGetLastError();
}

}  // namespace jarq
