// Bounded Babai proposal and acceptance for group i of every active row
// (Sec. 3.3.2, Eqs. conditional_residual, group_bils, group_qr,
// babai_update; App. E "Small scales").
//
// One warp per output row; lane owns the NT = g/32 consecutive coordinates
// l = NT*lane .. NT*lane + NT - 1.  The group factor L_i = R_i^T is staged in
// shared memory.
//
// The recursion is evaluated relative to the row's current codes q.  The
// target y = R_i^{-T} (H r)_i / s is formed in double-float as
// (Pt_i - T_i) / s: Pt_i = R_i^{-T} (H w)_i from the folded target projection
// and T_i = sum_h s_h R_i^{-T} H_ih c_h from the phase product (split-K
// partials), so that the cancellation of H's low-rank part costs no
// precision.  Then
//     v = R_i^{-T} [(H r)_i + s H_ii c] / s = y + R_i c,   c = q - z,
// so the pre-round value of Eq. babai_update is
//     z + x_l = q_l + (y_l - sum_{h>l} R_lh Delta_h) / R_ll,
// Delta_h = q^cand_h - q_h.  The running vector u = y - R Delta changes only
// where Delta != 0.  The back substitution scans h = g-1 .. 0: the lane that
// owns coordinate h rounds it, the change is broadcast, and only when it is
// non-zero do the coordinates below take the column update (a warp-uniform
// branch).  A row none of whose codes would change at u = y has no change
// at all (the first coordinate's value is final and unchanged, and so on
// down) and skips the scan.
//
// The change of the group objective (Eq. group_bils) is
// dF = s^2 (||R Delta - y||^2 - ||y||^2) = s^2 sum_l (a_l - y_l)(a_l + y_l)
// with a_l = R_ll Delta_l - u_l, exactly zero for an unchanged proposal.  A
// proposal is kept iff it changes a code, dF is finite and dF < 0.
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
    int row0, row1;              // rows [row0, row1) of this launch
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
    // partials are read and before the codes it reads are rewritten: each
    // thread waits for it just before reading the partials (the loads of a
    // row's flag, scale, zero point and Pt slice, which the phase product
    // does not write, come first).  The next grid is released only after
    // the wait: by then every grid before this one has completed, so the
    // next phase product may read the codes of the groups this step leaves
    // alone before its own wait.
    bool waited = false;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
    const int l0 = NT * lane;
    const int col0 = a.i * g;
    float rd[NT];
    load_vec<NT>(rdiag + l0, rd);
    for (int j = a.row0 + blockIdx.x * nwarps + wid; j < a.row1; j += gridDim.x * nwarps) {
        // the row's flag, scale and zero point, and this lane's slice of the
        // folded projection Pt_i, are loaded together
        const size_t off = (size_t)j * d + col0;
        const int act = a.active[j];
        const float s = a.S[(size_t)j * G + a.i];
        const int z = a.Z[(size_t)j * G + a.i];
        float y[NT], yl[NT];
        load_vec<NT>(a.pt_hi + off + l0, y);
        load_vec<NT>(a.pt_lo + off + l0, yl);
        if (!act) continue;
        if (!(fabsf(s) > a.eps)) continue;  // small-scale skip (also NaN)
        // s y = Pt_i - sum_sp T_sp, in double-float
        if (!waited) {
            tc::pdl_wait();
            tc::pdl_launch_dependents();
            waited = true;
        }
        for (int sp = 0; sp < a.nsplit; ++sp) {
            float th[NT], tl[NT];
            const size_t o = ((size_t)sp * a.rv.p_pad + j) * g + l0;
            load_vec<NT>(a.t_hi + o, th);
            load_vec<NT>(a.t_lo + o, tl);
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                const float sm = y[t] - th[t];
                const float bb = sm - y[t];
                const float e = (y[t] - (sm - bb)) + (-th[t] - bb);
                y[t] = sm;
                yl[t] += e - tl[t];
            }
        }
#pragma unroll
        for (int t = 0; t < NT; ++t) y[t] += yl[t];
        float qc[NT], qn[NT];   // current and proposed codes (small integers, exact)
        {
            uint32_t packed = 0;
            if constexpr (NT == 4) {
                packed = *reinterpret_cast<const uint32_t *>(a.Q + off + l0);
            } else {
                packed = *reinterpret_cast<const uint16_t *>(a.Q + off + l0);
            }
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                qc[t] = (float)((packed >> (8 * t)) & 0xFFu);
                qn[t] = qc[t];
            }
        }
        // y = R^{-T} (H r)_i / s
        float u[NT];
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            y[t] = y[t] / s;
            u[t] = y[t];
        }
        // back substitution (Eq. babai_update).  Rounding to the nearest
        // even integer adds and subtracts 1.5 * 2^23 (exact for |x| < 2^22;
        // beyond that the clamp to [0, qmax] gives the same code as rintf).
        const float qmaxf = (float)a.qmax;
        constexpr float kRound = 12582912.0f;      // 1.5 * 2^23
        bool any = false;
        // does any code change at u = y?
        int nchg = 0;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            const float x = fmaf(u[t], rd[t], qc[t]);
            const float r = __fsub_rn(__fadd_rn(x, kRound), kRound);
            nchg += fminf(fmaxf(r, 0.f), qmaxf) != qc[t];
        }
        if (__any_sync(0xffffffffu, nchg != 0)) {
            // descending scan (Eq. babai_update), coordinate h = NT L + t
            for (int L = 31; L >= 0; --L) {
#pragma unroll
                for (int t = NT - 1; t >= 0; --t) {
                    const int h = NT * L + t;
                    float dq = 0.f;
                    if (lane == L) {
                        const float x = fmaf(u[t], rd[t], qc[t]);
                        const float r = __fsub_rn(__fadd_rn(x, kRound), kRound);
                        const float q = fminf(fmaxf(r, 0.f), qmaxf);
                        dq = q - qc[t];
                        qn[t] = q;
                    }
                    dq = __shfl_sync(0xffffffffu, dq, L);
                    if (dq != 0.f) {                      // warp-uniform
                        any = true;
                        float lr[NT];
                        load_vec<NT>(Lg + h * g + l0, lr);   // R[l'][h] for l' = l0..
#pragma unroll
                        for (int tt = 0; tt < NT; ++tt)
                            if (l0 + tt < h) u[tt] = fmaf(-lr[tt], dq, u[tt]);
                    }
                }
            }
        }
        if (!any) continue;
        float acc = 0.f;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            const float av = Lg[(l0 + t) * g + l0 + t] * (qn[t] - qc[t]) - u[t];
            acc = fmaf(av - y[t], av + y[t], acc);
        }
        for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        const float dF = s * s * acc;
        if (!(isfinite(dF) && dF < 0.f)) continue;
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            if (qn[t] != qc[t]) {
                const int l = l0 + t;
                const int qi = (int)qn[t];
                a.Q[off + l] = (uint8_t)qi;
                store_code(a.rv, j, col0 + l, qi - z);
            }
        }
        if (lane == 0) a.accepted[j] += 1;
    }
}

}  // namespace

cudaError_t launch_babai(const float *t_hi, const float *t_lo, const float *pt_hi,
                         const float *pt_lo, int nsplit, const float *Lf, const float *S,
                         uint8_t *Q, const int32_t *Z, ResidualView rv, const int *active,
                         int *accepted, int *status, int p, int g, int i, int qmax, float eps,
                         int row0, int row1, cudaStream_t s, bool pdl) {
    if (row0 < 0 || row1 > p || row0 > row1) return cudaErrorInvalidValue;
    if (row0 == row1) return cudaSuccess;
    BabaiArgs a{t_hi, t_lo, pt_hi, pt_lo, nsplit, Lf, S, Q, Z, rv, active, accepted, status,
                p, g, i, qmax, eps, row0, row1};
    // one block per SM, one warp per row: spread the rows evenly over the SMs
    const int rows = row1 - row0;
    const int nsm = num_sms();
    int warps = (rows + nsm - 1) / nsm;
    if (warps > kMaxWarps) warps = kMaxWarps;
    if (warps < 1) warps = 1;
    int blocks = (rows + warps - 1) / warps;
    if (blocks > nsm) blocks = nsm;
    const size_t smem = ((size_t)g * g + g) * sizeof(float);
    cudaError_t e = cudaSuccess;
    if (g == 128) {
        e = cudaFuncSetAttribute(babai_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        e = launch_k(babai_kernel<4>, dim3(blocks), dim3(32 * warps), smem, s, pdl, a);
    } else if (g == 64) {
        e = cudaFuncSetAttribute(babai_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        e = launch_k(babai_kernel<2>, dim3(blocks), dim3(32 * warps), smem, s, pdl, a);
    } else {
        return cudaErrorInvalidValue;
    }
    return e;
}

}  // namespace jarq
