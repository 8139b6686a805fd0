// One Gauss-Seidel sweep over all G groups in one launch (Sec. 3.3.2; App. E
// "Order of updates"): for every row tile, the phase products T_i and the
// Babai proposals of groups i = 0 .. G-1 in order.
//
// Rows are independent (the objective separates over output rows, Sec. 3.3),
// so phase i+1 of a 128-row tile needs only phase i of the same tile: the
// tiles advance through their phases without any grid-wide barrier.  The
// four CTAs of a tile form a thread-block cluster; each computes one part of
// the phase product
//     T_i = sum_h s_h Ht_ih c_h          (Eq. conditional_residual, folded)
// -- g/64 column parts of group i times 4/(g/64) parts of the K range --
// exactly as the per-phase product kernel does (integer digit planes of the
// folded rows Ht in fp16, exact tensor-core digit sums, double-float
// combine), and writes its double-float partial to global memory.  A
// cluster barrier makes the partials visible; then each CTA runs the Babai
// proposal and acceptance (babai_row.cuh) for its 32 rows of the tile, with
// the group factor L_i staged in shared memory by one bulk copy, writes the
// accepted codes to Q and to the fp16 code plane, and a second cluster
// barrier makes those codes visible to the next phase's tensor-map loads.
//
// One CTA (576 threads):
//   warp 0       TMA producer (code tiles, digit tiles, the group factor)
//   warp 1       TMEM allocation and the single-thread MMA issuer
//   warps 2..17  drain (digit sums -> double-float partial), then Babai,
//                two rows per warp with interleaved back substitutions
// Three 48 KB pipeline stages and the 64 KB group factor fit the shared
// memory of one SM; the 512 TMEM columns hold two 4-plane accumulators.
//
// Every wait on an mbarrier is bounded; on a timeout the CTA stops issuing
// work, keeps arriving at the cluster barriers of the remaining phases (so
// that no CTA of its cluster waits forever), drains its own copies and MMAs
// and reports JARQ_ERR_TIMEOUT through the status word.
#include <cmath>

#include "babai_row.cuh"
#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kTileA = 128 * 64 * 2;   // codes: 128 rows x 64 K, fp16
constexpr int kTileB = 64 * 64 * 2;    // one digit plane: 64 rows of Ht x 64 K
constexpr int kStage = kTileA + 4 * kTileB;
constexpr int kStages = 3;
constexpr int kCluster = 4;            // CTAs per row tile
constexpr int kLBytes = 128 * 128 * 4; // group factor, float32, g = 128 at most
constexpr int kBarOff = kStages * kStage + kLBytes;
constexpr int kSmem = 1024 + kBarOff + 256;
constexpr uint32_t kIdesc = tc::idesc_f16_f32(128, 256);
constexpr int kDrainWarps = 16;
constexpr int kThreads = 32 * (2 + kDrainWarps);

struct SweepArgs {
    float *t_hi, *t_lo;           // [nks][p_pad][g] partials of T_i
    const float *pt_hi, *pt_lo;   // [p][d] folded target projection
    const float *Lf;              // [G][g][g] L_i = R_i^T
    const float *S;               // [p][G]
    const int *expoT;             // [G][G] block exponents of Ht
    uint8_t *Q;                   // [p][d]
    const int32_t *Z;             // [p][G]
    __half *cplane;               // [p_pad][d_pad]
    const int *active;
    int *accepted;
    int *status;
    int p, p_pad, d, d_pad, G, qmax, nks, seg;
    float eps, round_c;
};

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

template <int NT>
__global__ void __launch_bounds__(kThreads, 1)
    sweep_kernel(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapT,
                 SweepArgs a) {
    constexpr int g = 32 * NT;
    constexpr int ncol = g / 64;            // column parts of a group
    constexpr int nkc = g / 64;             // 64-wide K chunks per group
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float *Lg = (float *)(smem + kStages * kStage);
    uint64_t *bars = (uint64_t *)(smem + kBarOff);
    uint32_t *tmem_slot = (uint32_t *)(bars + 2 * kStages + 6);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    int *consumed = (int *)(tmem_slot + 2);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rank = (int)tc::cluster_ctarank();
    const int cpart = rank % ncol, kpart = rank / ncol;
    const int j0 = (blockIdx.x / kCluster) * 128;
    const int h0 = kpart * a.seg;
    const int nseg = max(0, min(a.G, h0 + a.seg) - h0);
    const int nchunks = nseg * nkc;

    auto full = [&](int s) { return tc::smem_u32(bars + s); };
    auto empty = [&](int s) { return tc::smem_u32(bars + kStages + s); };
    auto afull = [&](int b) { return tc::smem_u32(bars + 2 * kStages + b); };
    auto aempty = [&](int b) { return tc::smem_u32(bars + 2 * kStages + 2 + b); };
    const uint32_t lbar = tc::smem_u32(bars + 2 * kStages + 4);
    const uint32_t done = tc::smem_u32(bars + 2 * kStages + 5);
    auto tileA = [&](int s) { return tc::smem_u32(smem + s * kStage); };
    auto tileB = [&](int s, int t) { return tc::smem_u32(smem + s * kStage + kTileA + t * kTileB); };

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(full(s), 1);
            tc::mbar_init(empty(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::mbar_init(afull(b), 1);
            tc::mbar_init(aempty(b), kDrainWarps);
        }
        tc::mbar_init(lbar, 1);
        tc::mbar_init(done, 1);
        *abort_flag = 0;
        *consumed = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(tc::smem_u32(tmem_slot), 512);
        tc::tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tc::prefetch_tmap(&mapC);
        tc::prefetch_tmap(&mapT);
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // scales, active rows and codes come from the preceding kernels
    tc::pdl_wait();
    tc::pdl_launch_dependents();

    const BabaiRowArgs ra{a.t_hi, a.t_lo, a.pt_hi, a.pt_lo, a.nks, a.S, a.Q, a.Z, a.cplane,
                          a.active, a.accepted, a.p_pad, a.d, a.d_pad, g, a.G, a.qmax, a.eps};
    int cp = 0;               // producer: chunks issued
    int nl = 0;               // producer: group-factor copies issued
    int cm = 0, um = 0;       // MMA issuer: chunks consumed, accumulator units
    int ud = 0;               // drain: accumulator units drained

    for (int i = 0; i < a.G; ++i) {
        if (warp == 0 && lane == 0) {
            // ---------------- producer
            if (!*abort_flag) {
                // the group factor of this phase; the buffer is free, the
                // previous phase's Babai ended before the last cluster barrier
                tc::fence_proxy_async_smem();
                tc::mbar_expect_tx(lbar, (uint32_t)(g * g * sizeof(float)));
                tc::bulk_load(tc::smem_u32(Lg), a.Lf + (size_t)i * g * g, g * g * sizeof(float),
                              lbar);
                ++nl;
                // codes written by the previous phase, before the tensor-map loads
                tc::fence_proxy_async_global();
            }
            const int m0 = i * g + cpart * 64;    // first row of Ht (output column)
            for (int c = 0; c < nchunks && !*abort_flag; ++c) {
                const int s = cp % kStages;
                if (!tc::mbar_wait(empty(s), ((cp / kStages) & 1) ^ 1)) {
                    *abort_flag = 1;
                    break;
                }
                const int kx = h0 * g + c * 64;
                tc::mbar_expect_tx(full(s), kStage);
                tc::tma_load_2d(tileA(s), &mapC, full(s), kx, j0);
#pragma unroll
                for (int t = 0; t < 4; ++t)
                    tc::tma_load_2d(tileB(s, t), &mapT, full(s), kx, t * a.d_pad + m0);
                ++cp;
            }
        } else if (warp == 1 && lane == 0) {
            // ---------------- MMA issuer: one accumulator unit per group h
            for (int u = 0; u < nseg && !*abort_flag; ++u) {
                const int b = um & 1;
                if (!tc::mbar_wait(aempty(b), ((um >> 1) & 1) ^ 1)) {
                    *abort_flag = 1;
                    break;
                }
                tc::tc_fence_after();
                bool ok = true;
                for (int kc = 0; kc < nkc; ++kc) {
                    const int s = cm % kStages;
                    if (!tc::mbar_wait(full(s), (cm / kStages) & 1) || *abort_flag) {
                        *abort_flag = 1;
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
#pragma unroll
                    for (int sub = 0; sub < 4; ++sub) {
                        const uint64_t ad = tc::sdesc_sw128(tileA(s)) + 2 * sub;
                        const uint64_t bd = tc::sdesc_sw128(tileB(s, 0)) + 2 * sub;
                        tc::mma_bf16(tmem + b * 256, ad, bd, kIdesc, (kc | sub) != 0);
                    }
                    tc::mma_commit(empty(s));
                    ++cm;
                }
                if (!ok) break;
                tc::mma_commit(afull(b));
                ++um;
            }
        } else if (warp >= 2) {
            // ---------------- drain: digits -> double-float x s_h 2^(E - 9) -> partial
            const int q = warp & 3, cq = (warp - 2) >> 2;    // lane quarter, 16-column quarter
            const int row = j0 + 32 * q + lane;
            float hi[16], lo[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                hi[e] = 0.f;
                lo[e] = 0.f;
            }
            bool ok = __all_sync(0xffffffffu, !*abort_flag);
            const float *srow = a.S + (size_t)min(row, a.p - 1) * a.G;
            const int *erow = a.expoT + (size_t)i * a.G;
            float s_next = nseg > 0 ? srow[h0] : 0.f;
            int e_next = nseg > 0 ? erow[h0] : 0;
            for (int u = 0; u < nseg && ok; ++u) {
                const int b = ud & 1, h = h0 + u;
                const float s_cur = row < a.p ? s_next : 0.f;
                const int e_cur = e_next;
                if (u + 1 < nseg) {
                    s_next = srow[h + 1];
                    e_next = erow[h + 1];
                }
                bool w = tc::mbar_wait(afull(b), (ud >> 1) & 1);
                w = __shfl_sync(0xffffffffu, w && !*abort_flag, 0);
                tc::tc_fence_after();
                if (!w) {
                    ok = false;
                    *abort_flag = 1;
                    break;
                }
                const float scale = ldexpf(s_cur, e_cur - 9);
                const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + b * 256 + cq * 16;
#pragma unroll
                for (int cc = 0; cc < 16; cc += 8) {
                    uint32_t v0[8], v1[8], v2[8], v3[8];
                    tc::tmem_ld8(base + 0 * 64 + cc, v0);
                    tc::tmem_ld8(base + 1 * 64 + cc, v1);
                    tc::tmem_ld8(base + 2 * 64 + cc, v2);
                    tc::tmem_ld8(base + 3 * 64 + cc, v3);
                    tc::tmem_wait_ld();
                    if (cc == 8) {
                        // every digit sum of this group is in registers
                        tc::tc_fence_before();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(aempty(b));
                    }
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        // D_0 + D_1 2^-10 exactly as (vh, vl) (the digit sums
                        // are integers, |D_0| <= 128 qmax 512): t = D_1 2^-10
                        // rounded to a multiple of 2^-k, k chosen on the host
                        // so that |D_0 + t| < 2^(24-k); D_2, D_3 enter the
                        // low part.
                        float s2, e2;
                        const float d1 = __uint_as_float(v1[e]);
                        const float tq = __fsub_rn(__fmaf_rn(d1, 0x1p-10f, a.round_c), a.round_c);
                        const float vh = __fadd_rn(__uint_as_float(v0[e]), tq);
                        float vl = __fmaf_rn(d1, 0x1p-10f, -tq);
                        vl = fmaf(__uint_as_float(v2[e]), 0x1p-20f, vl);
                        vl = fmaf(__uint_as_float(v3[e]), 0x1p-30f, vl);
                        const float ph = vh * scale;
                        const float pe = fmaf(vh, scale, -ph);
                        two_sum(hi[cc + e], ph, s2, e2);
                        hi[cc + e] = s2;
                        lo[cc + e] += e2 + fmaf(vl, scale, pe);
                    }
                }
                ++ud;
            }
            if (ok && row < a.p) {
                const size_t o = ((size_t)kpart * a.p_pad + row) * g + cpart * 64 + cq * 16;
#pragma unroll
                for (int e = 0; e < 16; e += 4) {
                    float x[4], y[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) two_sum(hi[e + k], lo[e + k], x[k], y[k]);
                    *reinterpret_cast<float4 *>(a.t_hi + o + e) = make_float4(x[0], x[1], x[2], x[3]);
                    *reinterpret_cast<float4 *>(a.t_lo + o + e) = make_float4(y[0], y[1], y[2], y[3]);
                }
            }
        }
        __syncwarp();
        // the partials of every CTA of the tile are in global memory
        tc::cluster_sync();
        if (warp >= 2) {
            // ---------------- Babai for this CTA's 32 rows of the tile
            bool ok = !*abort_flag && tc::mbar_wait(lbar, i & 1);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) {
                *abort_flag = 1;
            } else {
                float rd[NT], dg[NT], Rl[NT][NT];
                babai_lane_factor<NT>(Lg, lane, rd, dg, Rl);
                const int j = j0 + 32 * rank + 2 * (warp - 2);
                const int js[2] = {j < a.p ? j : -1, j + 1 < a.p ? j + 1 : -1};
                babai_rows<NT, 2>(ra, js, i, Lg, rd, dg, Rl, lane);
            }
            // the accepted codes reach the next phase's tensor-map loads
            tc::fence_proxy_async_global();
        }
        __syncwarp();
        tc::cluster_sync();
    }

    // ---------------- teardown: nothing of this CTA may be in flight
    if (warp == 1 && lane == 0) {
        tc::mma_commit(done);
        if (!tc::mbar_wait(done, 0)) *abort_flag = 1;
        *consumed = cm;
    }
    __syncthreads();
    if (warp == 0 && lane == 0) {
        // copies issued but never consumed (after a timeout)
        for (int c = *consumed; c < cp; ++c)
            if (!tc::mbar_wait(full(c % kStages), (c / kStages) & 1)) *abort_flag = 1;
        if (nl > 0 && !tc::mbar_wait(lbar, (nl - 1) & 1)) *abort_flag = 1;
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, ST_TIMEOUT);
}

}  // namespace

// Parts of the K range of the sweep's phase products: the four CTAs of a
// row tile are (g/64 column parts) x (K parts).
int sweep_k_parts(int g) { return kCluster / (g / 64); }

cudaError_t launch_sweep(const CUtensorMap &mapC, const CUtensorMap &mapT, float *t_hi,
                         float *t_lo, const float *pt_hi, const float *pt_lo, const float *Lf,
                         const float *S, const int *expoT, uint8_t *Q, const int32_t *Z,
                         __half *cplane, const int *active, int *accepted, int *status, int p,
                         int p_pad, int d, int d_pad, int g, int G, int qmax, float eps,
                         cudaStream_t s) {
    if (qmax < 1 || qmax > 255 || (g != 64 && g != 128)) return cudaErrorInvalidValue;
    const int nks = sweep_k_parts(g);
    const int seg = (G + nks - 1) / nks;
    // quantum 2^-k of the exact digit split: the largest k with
    // 128 qmax 512 + 2^14 <= 2^(24-k)
    const double bound = 128.0 * qmax * 512.0 + 16384.0;
    int kq = 0;
    while (kq < 7 && bound <= std::ldexp(1.0, 24 - (kq + 1))) ++kq;
    const float round_c = (float)std::ldexp(1.5, 23 - kq);
    SweepArgs a{t_hi, t_lo, pt_hi, pt_lo, Lf, S, expoT, Q, Z, cplane, active, accepted, status,
                p, p_pad, d, d_pad, G, qmax, nks, seg, eps, round_c};
    const dim3 grid((p_pad / 128) * kCluster);
    if (g == 128) {
        static std::atomic<unsigned long long> attr_done{0};
        const cudaError_t e = set_max_dynamic_smem((const void *)sweep_kernel<4>, kSmem, attr_done);
        if (e != cudaSuccess) return e;
        return launch_pdl_cluster(sweep_kernel<4>, grid, dim3(kThreads), (size_t)kSmem, s,
                                  kCluster, mapC, mapT, a);
    }
    static std::atomic<unsigned long long> attr_done{0};
    const cudaError_t e = set_max_dynamic_smem((const void *)sweep_kernel<2>, kSmem, attr_done);
    if (e != cudaSuccess) return e;
    return launch_pdl_cluster(sweep_kernel<2>, grid, dim3(kThreads), (size_t)kSmem, s, kCluster,
                              mapC, mapT, a);
}

}  // namespace jarq
