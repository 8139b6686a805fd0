// Per-row reduction of the full residual product H r (tensor cores):
// F_j = r_j^T (H r_j) (Eq. bbmils_columns) and the scale gradient
// g_j[i] = c_i^T (H r_j)_i, the right-hand side of the normal equations of
// Eq. scale_normal_equations written for the increment of the scales.
#include "jarq_internal.cuh"

namespace jarq {
namespace {


// Per row (one warp): F_j = r_j . (H r_j) in float64 and the scale gradient
// g_j[i] = c_i . (H r_j)_i, c = q - z.
__global__ void grad_kernel(const uint8_t *__restrict__ Q, const int32_t *__restrict__ Z,
                            const float *__restrict__ r, const float *__restrict__ Hr,
                            double *__restrict__ gvec, double *__restrict__ F, int p, int d,
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
        if (lane == 0 && gvec) gvec[(size_t)warp * G + i] = gi;
    }
    for (int o = 16; o; o >>= 1) fs += __shfl_xor_sync(0xffffffffu, fs, o);
    if (lane == 0) F[warp] = fs;
}

}  // namespace

cudaError_t launch_grad(const uint8_t *Q, const int32_t *Z, const float *r, const float *Hr,
                        double *gvec, double *F, int p, int d, int g, cudaStream_t s) {
    grad_kernel<<<(p * 32 + 255) / 256, 256, 0, s>>>(Q, Z, r, Hr, gvec, F, p, d, g);
    return cudaGetLastError();
}

}  // namespace jarq
