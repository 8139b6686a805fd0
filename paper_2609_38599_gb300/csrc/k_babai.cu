// Per-phase Babai kernel: the bounded Babai proposal and acceptance of
// babai_row.cuh for group i of every active row, one warp per row, the group
// factor L_i staged in shared memory by one bulk copy.
#include "babai_row.cuh"
#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kMaxWarps = 32;   // warps per block (one row each) at most

struct BabaiArgs {
    const float *t_hi, *t_lo;    // [nsplit][p_pad][g] split-K partials of T_i
    const float *pt_hi, *pt_lo;  // [p][d] folded target projection Pt
    int nsplit;
    const float *Lf;
    const float *S;
    uint8_t *Q;
    const int32_t *Z;
    ResidualView rv;
    const int *active;
    int *accepted;
    int *status;
    int p, g, i, qmax;
    float eps;
};

template <int NT>
__global__ void __launch_bounds__(32 * kMaxWarps) babai_kernel(BabaiArgs a) {
    constexpr int g = 32 * NT;
    extern __shared__ __align__(16) float smem[];
    float *Lg = smem;                 // [g][g] lower factor of group i
    float *rdiag = Lg + g * g;        // [g] 1 / R_ll
    __shared__ uint64_t bar;
    __shared__ int load_ok;
    const int d = a.rv.d, G = d / g;
    // group factor of group i: one bulk copy (it does not depend on the
    // previous kernel, so it overlaps that kernel's tail under programmatic
    // launch)
    if (threadIdx.x == 0) {
        tc::mbar_init(tc::smem_u32(&bar), 1);
        tc::fence_barrier_init();
        tc::mbar_expect_tx(tc::smem_u32(&bar), (uint32_t)(g * g * sizeof(float)));
        tc::bulk_load(tc::smem_u32(Lg), a.Lf + (size_t)a.i * g * g, g * g * sizeof(float),
                      tc::smem_u32(&bar));
        load_ok = tc::mbar_wait(tc::smem_u32(&bar), 0) ? 1 : 0;
    }
    __syncthreads();
    if (!load_ok) {
        if (threadIdx.x == 0) atomicOr(a.status, ST_TIMEOUT);
        return;
    }
    for (int l = threadIdx.x; l < g; l += blockDim.x) rdiag[l] = 1.0f / Lg[l * g + l];
    __syncthreads();
    // the phase product (previous kernel) must be complete before its
    // partials are read and before the residual it reads is rewritten
    tc::pdl_wait();
    tc::pdl_launch_dependents();
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int l0 = NT * lane;
    float rd[NT];
    load_vec<NT>(rdiag + l0, rd);
    const BabaiRowArgs ra{a.t_hi, a.t_lo, a.pt_hi, a.pt_lo, a.nsplit, a.S, a.Q, a.Z,
                          a.rv.cplane, a.active, a.accepted, a.rv.p_pad, d, a.rv.d_pad,
                          g, G, a.qmax, a.eps};
    for (int j = blockIdx.x * nwarps + wid; j < a.p; j += gridDim.x * nwarps)
        babai_row<NT>(ra, j, a.i, Lg, rd, lane);
}

}  // namespace

cudaError_t launch_babai(const float *t_hi, const float *t_lo, const float *pt_hi,
                         const float *pt_lo, int nsplit, const float *Lf, const float *S,
                         uint8_t *Q, const int32_t *Z, ResidualView rv, const int *active,
                         int *accepted, int *status, int p, int g, int i, int qmax, float eps,
                         cudaStream_t s) {
    BabaiArgs a{t_hi, t_lo, pt_hi, pt_lo, nsplit, Lf, S, Q, Z, rv, active, accepted, status,
                p, g, i, qmax, eps};
    // one block per SM, one warp per row: spread the rows evenly over the SMs
    const int nsm = num_sms();
    int warps = (p + nsm - 1) / nsm;
    if (warps > kMaxWarps) warps = kMaxWarps;
    if (warps < 1) warps = 1;
    int blocks = (p + warps - 1) / warps;
    if (blocks > nsm) blocks = nsm;
    const size_t smem = ((size_t)g * g + g) * sizeof(float);
    cudaError_t e = cudaSuccess;
    if (g == 128) {
        e = cudaFuncSetAttribute(babai_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        e = launch_pdl(babai_kernel<4>, dim3(blocks), dim3(32 * warps), smem, s, a);
    } else if (g == 64) {
        e = cudaFuncSetAttribute(babai_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        e = launch_pdl(babai_kernel<2>, dim3(blocks), dim3(32 * warps), smem, s, a);
    } else {
        return cudaErrorInvalidValue;
    }
    return e;
}

}  // namespace jarq
