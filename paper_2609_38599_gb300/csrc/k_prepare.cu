// Hessian preparation: symmetrisation, per-group Cholesky factors and the
// folded operand of the sweep's residual products.
//
// Sec. 3.3.2, Eq. group_qr: each group's factor R_i (A_i = U_i R_i) is
// computed once per layer and reused for every output row and iteration.
// With H = A^T A, R_i^T R_i = H_ii, so R_i is taken as the upper Cholesky
// factor of H_ii (equal to the QR factor up to row signs, to which the
// Babai recursion is invariant).  The factor and its inverse are computed in
// float64 in shared memory:
//   Lf[i]   = L_i = R_i^T          (lower, row-major: Lf[l][m] = R_i[m][l]), float32
//   Rinv[i] = R_i^{-1}             (upper, row-major), float64
// The Babai target of Eq. babai_update needs y = R_i^{-T} (H r)_i / s.  The
// rows H_i of group i are dominated by the low-rank part of H, which R_i^{-T}
// cancels: forming (H r)_i first and applying R_i^{-T} afterwards amplifies
// the product's rounding by up to sqrt(cond(H_ii)).  The sweep therefore
// works with the folded rows
//   Ht[grp i, :] = R_i^{-T} H[grp i, :]
// computed here once, in double-float (hi + lo) from the float64 inverse.
#include "jarq_internal.cuh"

namespace jarq {
namespace {

// out = (H + H^T)/2 + nu2 I, through 32x32 shared-memory tiles, plus its
// exact three-plane bf16 split (planes [3][d_pad][d_pad], pitch d_pad).
__global__ void symmetrize_kernel(const float *__restrict__ H, float *__restrict__ Hs,
                                  __nv_bfloat16 *__restrict__ planes, int d, int d_pad,
                                  float nu2) {
    __shared__ float tile[32][33];
    const int bx = blockIdx.x * 32, by = blockIdx.y * 32;
    const int tx = threadIdx.x, ty = threadIdx.y;  // 32 x 8
    for (int yy = ty; yy < 32; yy += 8) {
        int row = bx + yy, col = by + tx;  // transposed block
        tile[yy][tx] = (row < d && col < d) ? H[(size_t)row * d + col] : 0.f;
    }
    __syncthreads();
    for (int yy = ty; yy < 32; yy += 8) {
        int row = by + yy, col = bx + tx;
        if (row < d && col < d) {
            float v = 0.5f * (H[(size_t)row * d + col] + tile[tx][yy]);
            if (row == col) v += nu2;
            Hs[(size_t)row * d + col] = v;
            __nv_bfloat16 a, b, c;
            split3(v, a, b, c);
            const size_t plane = (size_t)d_pad * d_pad, off = (size_t)row * d_pad + col;
            planes[off] = a;
            planes[plane + off] = b;
            planes[2 * plane + off] = c;
        }
    }
}

// One block per group: float64 Cholesky of H_ii in shared memory, then an
// in-place inverse of the lower factor.
__global__ void group_factor_kernel(const float *__restrict__ Hs, float *__restrict__ Lf,
                                    double *__restrict__ L64, double *__restrict__ Rinv, int d,
                                    int g, int *status) {
    extern __shared__ double smem[];
    const int ld = g + 1;
    double *A = smem;               // [g][g+1]
    double *tmp = smem + g * ld;    // [g]
    __shared__ int failed;
    const int grp = blockIdx.x;
    const int base = grp * g;
    const int tid = threadIdx.x, nt = blockDim.x;
    if (tid == 0) failed = 0;
    for (int idx = tid; idx < g * g; idx += nt) {
        int a = idx / g, b = idx % g;
        A[a * ld + b] = (double)Hs[(size_t)(base + a) * d + base + b];
    }
    __syncthreads();
    // right-looking Cholesky, lower triangle
    for (int k = 0; k < g; ++k) {
        if (tid == 0) {
            double piv = A[k * ld + k];
            if (!(piv > 0.0) || !isfinite(piv)) {
                failed = 1;
            } else {
                A[k * ld + k] = sqrt(piv);
            }
        }
        __syncthreads();
        if (failed) break;
        const double lkk = A[k * ld + k];
        for (int a = k + 1 + tid; a < g; a += nt) A[a * ld + k] /= lkk;
        __syncthreads();
        const int n = g - k - 1;
        for (int idx = tid; idx < n * n; idx += nt) {
            int a = k + 1 + idx / n, b = k + 1 + idx % n;
            if (b <= a) A[a * ld + b] -= A[a * ld + k] * A[b * ld + k];
        }
        __syncthreads();
    }
    if (failed) {
        if (tid == 0) atomicOr(status, ST_NOT_SPD);
        return;
    }
    float *Lo = Lf + (size_t)grp * g * g;
    double *Ld = L64 + (size_t)grp * g * g;
    for (int idx = tid; idx < g * g; idx += nt) {
        int a = idx / g, b = idx % g;
        Lo[idx] = (b <= a) ? (float)A[a * ld + b] : 0.f;
        Ld[idx] = (b <= a) ? A[a * ld + b] : 0.0;
    }
    __syncthreads();
    // in-place inverse of the lower factor, columns from last to first:
    // Linv[j][j] = 1/L[j][j]; Linv[j+1:, j] = -Linv[j][j] * Linv[j+1:, j+1:] L[j+1:, j]
    for (int j = g - 1; j >= 0; --j) {
        for (int a = j + 1 + tid; a < g; a += nt) tmp[a] = A[a * ld + j];
        __syncthreads();
        const double inv_jj = 1.0 / A[j * ld + j];
        for (int a = j + 1 + tid; a < g; a += nt) {
            double acc = 0.0;
            for (int b = j + 1; b <= a; ++b) acc += A[a * ld + b] * tmp[b];
            A[a * ld + j] = -acc * inv_jj;
        }
        __syncthreads();
        if (tid == 0) A[j * ld + j] = inv_jj;
        __syncthreads();
    }
    // Rinv = (L^{-1})^T : Rinv[m][l] = Linv[l][m]
    double *Ri = Rinv + (size_t)grp * g * g;
    for (int idx = tid; idx < g * g; idx += nt) {
        int m = idx / g, l = idx % g;
        Ri[idx] = (l >= m) ? A[l * ld + m] : 0.0;
    }
}

// (s, e) with s + e = a + b exactly
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

// Ht[i g + a, k] = sum_{b <= a} Rinv_i[b][a] Hs[i g + b, k] for one group i
// (blockIdx.y) and 64 columns k (blockIdx.x): Rinv_i as float pairs (hi, lo)
// and the H tile in shared memory, double-float accumulation, written as the
// float pair (hi, lo) [d][d].
constexpr int kHtCols = 64;

__global__ void __launch_bounds__(256) htilde_kernel(const float *__restrict__ Hs,
                                                     const double *__restrict__ Rinv,
                                                     float *__restrict__ out_hi,
                                                     float *__restrict__ out_lo, int d, int g) {
    extern __shared__ float hsm[];
    float *rh = hsm;                   // [g][g] hi parts, Rinv[b][a] at b * g + a
    float *rl = rh + g * g;            // [g][g] lo parts
    float *ht = rl + g * g;            // [g][kHtCols] rows of H for this group
    const int i = blockIdx.y, k0 = blockIdx.x * kHtCols;
    const int tid = threadIdx.x;
    const double *Ri = Rinv + (size_t)i * g * g;
    for (int idx = tid; idx < g * g; idx += blockDim.x) {
        const double v = Ri[idx];
        const float hi = (float)v;
        rh[idx] = hi;
        rl[idx] = (float)(v - (double)hi);
    }
    for (int idx = tid; idx < g * kHtCols; idx += blockDim.x) {
        const int b = idx / kHtCols, kk = idx % kHtCols;
        ht[idx] = (k0 + kk < d) ? Hs[(size_t)(i * g + b) * d + k0 + kk] : 0.f;
    }
    __syncthreads();
    const int kk = tid % kHtCols, a0 = tid / kHtCols, astep = blockDim.x / kHtCols;
    for (int a = a0; a < g; a += astep) {
        float sh = 0.f, sl = 0.f;
        for (int b = 0; b <= a; ++b) {
            const float hv = ht[b * kHtCols + kk];
            const float r_hi = rh[b * g + a], r_lo = rl[b * g + a];
            const float m = r_hi * hv;
            float e = fmaf(r_hi, hv, -m);
            e = fmaf(r_lo, hv, e);
            float s2, e2;
            two_sum(sh, m, s2, e2);
            sh = s2;
            sl += e2 + e;
        }
        if (k0 + kk < d) {
            float s2, e2;
            two_sum(sh, sl, s2, e2);
            const size_t off = (size_t)(i * g + a) * d + k0 + kk;
            out_hi[off] = s2;
            out_lo[off] = e2;
        }
    }
}

}  // namespace

cudaError_t launch_symmetrize(const float *H, float *Hs, __nv_bfloat16 *Hplanes, int d, int d_pad,
                              float nu2, cudaStream_t s) {
    dim3 grid((d + 31) / 32, (d + 31) / 32), block(32, 8);
    symmetrize_kernel<<<grid, block, 0, s>>>(H, Hs, Hplanes, d, d_pad, nu2);
    return cudaGetLastError();
}

cudaError_t launch_group_factor(const float *Hs, float *Lf, double *L64, double *Rinv, int d,
                                int g, int *status, cudaStream_t s) {
    size_t smem = (size_t)(g * (g + 1) + g) * sizeof(double);
    cudaError_t e = cudaFuncSetAttribute(group_factor_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    group_factor_kernel<<<d / g, 256, smem, s>>>(Hs, Lf, L64, Rinv, d, g, status);
    return cudaGetLastError();
}

cudaError_t launch_htilde(const float *Hs, const double *Rinv, float *out_hi, float *out_lo,
                          int d, int g, cudaStream_t s) {
    const size_t smem = ((size_t)2 * g * g + (size_t)g * kHtCols) * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(htilde_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((d + kHtCols - 1) / kHtCols, d / g);
    htilde_kernel<<<grid, 256, smem, s>>>(Hs, Rinv, out_hi, out_lo, d, g);
    return cudaGetLastError();
}

}  // namespace jarq
