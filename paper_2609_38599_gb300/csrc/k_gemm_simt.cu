// CUDA-core contractions of the refinement path (float32, register tiled).
//
// All products read the symmetrised Hessian H (ldb = d) as the right
// operand with a 64 x 128 output tile per block:
//   hr_full   H r_j for every row (objective of Eq. bbmils_columns and the
//             scale gradient g_j[i] = c_i^T (H r_j)_i, i.e. the right-hand side
//             of the normal equations of Eq. scale_normal_equations written
//             for the increment of the scales)
//   gram      Gram_j[i,h] = c_i^T H_ih c_h      (Sec. 3.3.1, Eq. scale_design)
//   phase_hr  (H r_j)_i for one group i, split over K  (Eq. conditional_residual)
// The residual r = w - D_s (q - z) enters directly (no W H - H What
// cancellation).  Long K loops accumulate in 128-term chunks to bound float32
// error growth.
#include "jarq_internal.cuh"

namespace jarq {
namespace {

constexpr int BM = 64, BN = 128, BK = 16, NT = 256;

struct SmemTile {
    float As[BK][BM];
    float Bs[BK][BN];
};

struct DenseA {  // A[j][k] from a float32 row-major matrix
    const float *A;
    int lda;
    __device__ float operator()(int j, int k) const { return A[(size_t)j * lda + k]; }
};

struct CodeA {  // c[j][k] = q[j][k] - z[j][k / g]
    const uint8_t *Q;
    const int32_t *Z;
    int d, g, G;
    __device__ float operator()(int j, int k) const {
        return (float)((int)Q[(size_t)j * d + k] - Z[(size_t)j * G + k / g]);
    }
};

// acc[a][e] (+)= sum_{k in [kbeg,kend)} A[row0+ty*4+a][k] * B[k][col(e)],
// col(e) = n0 + (e < 4 ? tx*4+e : 64+tx*4+e-4), columns >= n_end read as 0.
template <class AL>
__device__ __forceinline__ void tile_product(float (&acc)[4][8], const AL &aload, int p,
                                             int row0, const float *__restrict__ B, int ldb,
                                             int n0, int n_end, int kbeg, int kend,
                                             SmemTile &sm) {
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    float ra[4], rb[8];
    auto load = [&](int k0) {
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            int e = tid + NT * t, row = e >> 4, kk = e & 15;
            int j = row0 + row, k = k0 + kk;
            ra[t] = (j < p && k < kend) ? aload(j, k) : 0.f;
        }
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            int e = tid + NT * t, kk = e >> 7, n = e & 127;
            int k = k0 + kk, col = n0 + n;
            rb[t] = (k < kend && col < n_end) ? B[(size_t)k * ldb + col] : 0.f;
        }
    };
    load(kbeg);
    for (int k0 = kbeg; k0 < kend; k0 += BK) {
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            int e = tid + NT * t;
            sm.As[e & 15][e >> 4] = ra[t];
        }
#pragma unroll
        for (int t = 0; t < 8; ++t) {
            int e = tid + NT * t;
            sm.Bs[e >> 7][e & 127] = rb[t];
        }
        __syncthreads();
        if (k0 + BK < kend) load(k0 + BK);
#pragma unroll
        for (int kk = 0; kk < BK; ++kk) {
            float4 a = *reinterpret_cast<const float4 *>(&sm.As[kk][ty * 4]);
            float4 b0 = *reinterpret_cast<const float4 *>(&sm.Bs[kk][tx * 4]);
            float4 b1 = *reinterpret_cast<const float4 *>(&sm.Bs[kk][64 + tx * 4]);
            float av[4] = {a.x, a.y, a.z, a.w};
            float bv[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
            for (int x = 0; x < 4; ++x)
#pragma unroll
                for (int y = 0; y < 8; ++y) acc[x][y] = fmaf(av[x], bv[y], acc[x][y]);
        }
        __syncthreads();
    }
}

__device__ __forceinline__ int col_of(int tx, int e) {
    return e < 4 ? tx * 4 + e : 64 + tx * 4 + (e - 4);
}

// Long-K product with chunked accumulation: tot = sum over 128-wide chunks.
template <class AL>
__device__ __forceinline__ void long_product(float (&tot)[4][8], const AL &aload, int p,
                                             int row0, const float *__restrict__ B, int ldb,
                                             int n0, int n_end, int kbeg, int kend,
                                             SmemTile &sm) {
#pragma unroll
    for (int x = 0; x < 4; ++x)
#pragma unroll
        for (int y = 0; y < 8; ++y) tot[x][y] = 0.f;
    for (int c0 = kbeg; c0 < kend; c0 += 128) {
        float acc[4][8];
#pragma unroll
        for (int x = 0; x < 4; ++x)
#pragma unroll
            for (int y = 0; y < 8; ++y) acc[x][y] = 0.f;
        tile_product(acc, aload, p, row0, B, ldb, n0, n_end, c0, min(kend, c0 + 128), sm);
#pragma unroll
        for (int x = 0; x < 4; ++x)
#pragma unroll
            for (int y = 0; y < 8; ++y) tot[x][y] += acc[x][y];
    }
}

__device__ __forceinline__ float reduce16(float v) {
    v += __shfl_xor_sync(0xffffffffu, v, 8);
    v += __shfl_xor_sync(0xffffffffu, v, 4);
    v += __shfl_xor_sync(0xffffffffu, v, 2);
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    return v;
}

__device__ __forceinline__ bool tile_has_active(const int *active, int p, int row0) {
    int mine = 0;
    if (threadIdx.x < BM && row0 + (int)threadIdx.x < p) mine = active[row0 + threadIdx.x];
    return __syncthreads_or(mine) != 0;
}

// C = A H for a float32 row-major A [p][d] (used with A = r).
__global__ void __launch_bounds__(NT) product_kernel(const float *__restrict__ A,
                                                     const float *__restrict__ Hs,
                                                     float *__restrict__ C, int p, int d) {
    __shared__ SmemTile sm;
    const int row0 = blockIdx.x * BM, n0 = blockIdx.y * BN;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float tot[4][8];
    long_product(tot, DenseA{A, d}, p, row0, Hs, d, n0, d, 0, d, sm);
#pragma unroll
    for (int x = 0; x < 4; ++x) {
        int j = row0 + ty * 4 + x;
        if (j >= p) continue;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            int col = n0 + col_of(tx, e);
            if (col < d) C[(size_t)j * d + col] = tot[x][e];
        }
    }
}

// Per row (one warp): F_j = r_j . (H r_j) in float64 and the scale gradient
// g_j[i] = c_i . (H r_j)_i, c = q - z.
__global__ void grad_kernel(const uint8_t *__restrict__ Q, const int32_t *__restrict__ Z,
                            const float *__restrict__ r, const float *__restrict__ Hr,
                            float *__restrict__ gvec, double *__restrict__ F, int p, int d,
                            int g) {
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    if (warp >= p) return;
    const int G = d / g;
    const size_t off = (size_t)warp * d;
    double fs = 0.0;
    for (int i = 0; i < G; ++i) {
        double gi = 0.0;
        const int z = Z[(size_t)warp * G + i];
        for (int m = lane; m < g; m += 32) {
            const size_t idx = off + (size_t)i * g + m;
            const double hv = (double)Hr[idx];
            gi += (double)((int)Q[idx] - z) * hv;
            fs += (double)r[idx] * hv;
        }
        for (int o = 16; o; o >>= 1) gi += __shfl_xor_sync(0xffffffffu, gi, o);
        if (lane == 0 && gvec) gvec[(size_t)warp * G + i] = (float)gi;
    }
    for (int o = 16; o; o >>= 1) fs += __shfl_xor_sync(0xffffffffu, fs, o);
    if (lane == 0) F[warp] = fs;
}

__global__ void __launch_bounds__(NT) phase_hr_kernel(const float *__restrict__ r,
                                                      const float *__restrict__ Hs,
                                                      const int *__restrict__ active,
                                                      float *__restrict__ hr, int p, int d, int g,
                                                      int grp) {
    __shared__ SmemTile sm;
    const int row0 = blockIdx.x * BM;
    if (!tile_has_active(active, p, row0)) return;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int split = blockIdx.y, nsplit = gridDim.y;
    const int kc = ((d + nsplit - 1) / nsplit + BK - 1) / BK * BK;
    const int kbeg = split * kc, kend = min(d, kbeg + kc);
    const int n0 = grp * g;
    float tot[4][8];
    long_product(tot, DenseA{r, d}, p, row0, Hs, d, n0, n0 + g, kbeg, kend, sm);
    float *out = hr + (size_t)split * p * g;
#pragma unroll
    for (int x = 0; x < 4; ++x) {
        int j = row0 + ty * 4 + x;
        if (j >= p) continue;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            int m = col_of(tx, e);
            if (m < g) out[(size_t)j * g + m] = tot[x][e];
        }
    }
}

__global__ void __launch_bounds__(NT) gram_kernel(const uint8_t *__restrict__ Q,
                                                  const int32_t *__restrict__ Z,
                                                  const float *__restrict__ Hs,
                                                  const int *__restrict__ active,
                                                  float *__restrict__ gram, int p, int d, int g) {
    __shared__ SmemTile sm;
    __shared__ float Ci[BM][BN + 4];
    const int G = d / g;
    const int row0 = blockIdx.x * BM, i = blockIdx.y;
    if (!tile_has_active(active, p, row0)) return;
    const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
    const CodeA code{Q, Z, d, g, G};
    for (int e = tid; e < BM * BN; e += NT) {
        int row = e / BN, m = e % BN, j = row0 + row;
        Ci[row][m] = (j < p && m < g) ? code(j, i * g + m) : 0.f;
    }
    __syncthreads();
    for (int h = 0; h < G; ++h) {
        float acc[4][8];
#pragma unroll
        for (int x = 0; x < 4; ++x)
#pragma unroll
            for (int y = 0; y < 8; ++y) acc[x][y] = 0.f;
        // D[j][m] = sum_{k in grp h} c[j][k] H[k][i g + m] = (c_h^T H_{h,i})[m]
        tile_product(acc, code, p, row0, Hs, d, i * g, i * g + g, h * g, h * g + g, sm);
#pragma unroll
        for (int x = 0; x < 4; ++x) {
            int row = ty * 4 + x, j = row0 + row;
            float part = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) part = fmaf(Ci[row][col_of(tx, e)], acc[x][e], part);
            part = reduce16(part);
            if (tx == 0 && j < p) gram[((size_t)j * G + i) * G + h] = part;
        }
    }
}

}  // namespace

cudaError_t launch_hr_full(const float *r, const float *Hs, float *Hr, int p, int d,
                          cudaStream_t s) {
    dim3 grid((p + BM - 1) / BM, (d + BN - 1) / BN);
    product_kernel<<<grid, NT, 0, s>>>(r, Hs, Hr, p, d);
    return cudaGetLastError();
}

cudaError_t launch_grad(const uint8_t *Q, const int32_t *Z, const float *r, const float *Hr,
                        float *gvec, double *F, int p, int d, int g, cudaStream_t s) {
    grad_kernel<<<(p * 32 + 255) / 256, 256, 0, s>>>(Q, Z, r, Hr, gvec, F, p, d, g);
    return cudaGetLastError();
}

cudaError_t launch_phase_hr(const float *r, const float *Hs, const int *active, float *hr,
                            int p, int d, int g, int i, cudaStream_t s) {
    dim3 grid((p + BM - 1) / BM, kSplitK);
    phase_hr_kernel<<<grid, NT, 0, s>>>(r, Hs, active, hr, p, d, g, i);
    return cudaGetLastError();
}

cudaError_t launch_gram(const uint8_t *Q, const int32_t *Z, const float *Hs, const int *active,
                        float *gram, int p, int d, int g, cudaStream_t s) {
    dim3 grid((p + BM - 1) / BM, d / g);
    gram_kernel<<<grid, NT, 0, s>>>(Q, Z, Hs, active, gram, p, d, g);
    return cudaGetLastError();
}

}  // namespace jarq
