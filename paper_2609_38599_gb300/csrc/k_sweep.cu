// One Gauss-Seidel sweep over all G groups in one launch (Sec. 3.3.2; App. E
// "Order of updates"): for every row tile, the phase products T_i and the
// bounded Babai proposals of groups i = 0 .. G-1 in order.
//
// Rows are independent (the objective separates over output rows, Sec. 3.3),
// so phase i+1 of a 128-row tile needs only phase i of the same tile: the
// tiles advance through their phases without any grid-wide barrier.  The
// four CTAs of a tile form a thread-block cluster; each computes one part of
// the phase product
//     T_i = sum_h s_h Ht_ih c_h          (Eq. conditional_residual, folded)
// -- g/64 column parts of group i times 4/(g/64) parts of the K range --
// from integer digit planes of the folded rows Ht (fp16, exact tensor-core
// digit sums, double-float combine) and writes its double-float partial to
// global memory.  Each CTA then forms the Babai targets
//     y = (Pt_i - T_i) / s_i = R_i^{-T} (H r)_i / s_i
// of its 32 rows of the tile from the partials of all four, and one Babai
// warp runs the proposal and acceptance of those 32 rows, one row per lane,
// while the product of the next phase proceeds.
//
// Overlap.  Group i's codes change only in phase i, so the product of phase
// i+1 needs phase i's result only for the K chunks of group i.  The CTA
// whose K range holds group i takes that group last in phase i+1, and its
// producer waits for the codes of all four Babai warps only before loading
// it; the other K chunks, and the other CTAs, go on meanwhile.
//
// One CTA (608 threads):
//   warp 0       TMA producer (code tiles, digit tiles)
//   warp 1       TMEM allocation and the single-thread MMA issuer
//   warps 2..17  drain: digit sums -> double-float partial; then the Babai
//                targets of two rows each, written to shared memory
//   warp 18      Babai: 32 rows, one per lane, back substitution by blocks
//                of 16 coordinates (its own factor R_i, bulk-copied)
// Cluster signals: two counters in every CTA's shared memory that each of
// the four CTAs increments once per phase (remote reductions with release
// semantics at cluster scope; readers poll with acquire): `pcnt` -- the
// partials of the phase are in global memory; `ccnt` -- the codes of the
// phase are in Q and the code plane.  Phase i is complete at 4 (i + 1).
// Counters, unlike barrier phases, may be waited for out of order: the
// producer waits only in the phases where it holds the pending group.
//
// Every wait is bounded; on a timeout the CTA stops issuing work, keeps
// arriving at the final cluster barrier (so no CTA of its cluster waits
// forever), drains its own copies and MMAs and reports JARQ_ERR_TIMEOUT.
#include <cmath>

#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kTileA = 128 * 64 * 2;   // codes: 128 rows x 64 K, fp16
constexpr int kTileB = 64 * 64 * 2;    // one digit plane: 64 rows of Ht x 64 K
constexpr int kStage = kTileA + 4 * kTileB;
constexpr int kStages = 3;
constexpr int kCluster = 4;            // CTAs per row tile
constexpr int kRows = 128 / kCluster;  // Babai rows per CTA (one per lane)
constexpr uint32_t kIdesc = tc::idesc_f16_f32(128, 256);
constexpr int kDrainWarps = 16;
constexpr int kBabaiWarp = 2 + kDrainWarps;
constexpr int kThreads = 32 * (kBabaiWarp + 1);

// Packed rows of R_i (upper triangular, g x g): row l holds columns
// 16 floor(l/16) .. g-1, so every row starts on a 64-byte boundary and a
// block of 16 columns is four aligned float4.
__host__ __device__ constexpr int rpk_row_off(int l, int g) {
    return 16 * ((l >> 4) * g - 8 * (l >> 4) * ((l >> 4) - 1)) + (l & 15) * (g - 16 * (l >> 4));
}
__host__ __device__ constexpr int rpk_size(int g) { return rpk_row_off(g, g); }

// shared memory (g = 128 sizes; g = 64 uses less of each)
constexpr int kOffRpk = kStages * kStage;
constexpr int kOffU = kOffRpk + rpk_size(128) * 4;
constexpr int kOffY = kOffU + 128 * kRows * 4;
constexpr int kOffC = kOffY + 128 * kRows * 4;
constexpr int kOffRd = kOffC + 32 * kRows * 4;
constexpr int kOffDg = kOffRd + 128 * 4;
constexpr int kOffRow = kOffDg + 128 * 4;         // s, z, live of the 32 rows
constexpr int kOffBar = kOffRow + 3 * kRows * 4;
constexpr int kSmem = 1024 + kOffBar + 256;
static_assert(kSmem <= 232448, "shared memory of one CTA");

struct SweepArgs {
    float *t_hi, *t_lo;           // [2][nks][p_pad][g] partials of T_i (two phases)
    const float *pt_hi, *pt_lo;   // [p][d] folded target projection
    const float *Rpk;             // [G][rpk_size(g)] packed factors R_i
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

// Group of K unit u of phase i for the CTA whose K range is [h0, h0 + nseg):
// when that range holds group i-1 (whose codes phase i-1 is still deciding),
// the units start after it and end with it.
__device__ __forceinline__ int unit_group(int u, int i, int h0, int nseg) {
    const int gp = i - 1;
    const int rot = (gp >= h0 && gp < h0 + nseg) ? gp - h0 + 1 : 0;
    int k = rot + u;
    if (k >= nseg) k -= nseg;
    return h0 + k;
}

// Smem index of coordinate l of Babai row r in the u and y arrays: [l][r],
// the row index XOR-ed with l/4 so that both the drain's writes (a row per
// warp, l across lanes) and the Babai warp's reads (l fixed, a row per lane)
// are free of bank conflicts.
__device__ __forceinline__ int uy_idx(int l, int r) { return l * kRows + (r ^ ((l >> 2) & 31)); }
// Word of the code array holding codes 4k .. 4k+3 of row r.
__device__ __forceinline__ int c_idx(int k, int r) { return k * kRows + (r ^ (k & 31)); }

template <int NT>
__global__ void __launch_bounds__(kThreads, 1)
    sweep_kernel(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapT,
                 SweepArgs a) {
    constexpr int g = 32 * NT;
    constexpr int ncol = g / 64;            // column parts of a group
    constexpr int nkc = g / 64;             // 64-wide K chunks per group
    constexpr int kRpk = rpk_size(g);
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float *Rs = (float *)(smem + kOffRpk);
    float *Ub = (float *)(smem + kOffU);
    float *Yb = (float *)(smem + kOffY);
    uint32_t *Cb = (uint32_t *)(smem + kOffC);
    float *Rd = (float *)(smem + kOffRd);
    float *Dg = (float *)(smem + kOffDg);
    float *rowS = (float *)(smem + kOffRow);
    int *rowZ = (int *)(rowS + kRows);
    int *rowLive = rowZ + kRows;
    uint64_t *bars = (uint64_t *)(smem + kOffBar);
    uint32_t *tmem_slot = (uint32_t *)(bars + 2 * kStages + 9);
    uint32_t *counters = tmem_slot + 4;   // pcnt, ccnt
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
    const uint32_t pcnt = tc::smem_u32(counters);       // partials, 4 per phase
    const uint32_t ccnt = tc::smem_u32(counters + 1);   // codes, 4 per phase
    const uint32_t ybar = tc::smem_u32(bars + 2 * kStages + 6);   // Babai targets, 16 warps
    const uint32_t lbar = tc::smem_u32(bars + 2 * kStages + 7);   // factor copy
    const uint32_t done = tc::smem_u32(bars + 2 * kStages + 8);
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
        counters[0] = 0;
        counters[1] = 0;
        tc::mbar_init(ybar, kDrainWarps);
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
    __syncwarp();
    // every CTA's barriers are initialised before any CTA arrives on them
    tc::cluster_sync();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // scales, active rows and codes come from the preceding kernels
    tc::pdl_wait();
    tc::pdl_launch_dependents();

    int cp = 0;               // producer: chunks issued
    int cm = 0;               // MMA issuer: chunks consumed
    int nl = 0;               // Babai warp: factor copies issued

    if (warp == 0 && lane == 0) {
        // ------------------------------------------------ producer
        for (int i = 0; i < a.G && !*abort_flag; ++i) {
            const int m0 = i * g + cpart * 64;    // first row of Ht (output column)
            const bool holds = i >= 1 && i - 1 >= h0 && i - 1 < h0 + nseg;
            for (int c = 0; c < nchunks; ++c) {
                const int u = c / nkc, kc = c % nkc;
                if (holds && u == nseg - 1 && kc == 0) {
                    // the last group is i-1: its codes from all four Babai warps
                    if (!tc::wait_count_cluster(ccnt, kCluster * i)) {
                        *abort_flag = 1;
                        break;
                    }
                    tc::fence_proxy_async_global();
                }
                const int s = cp % kStages;
                if (!tc::mbar_wait(empty(s), ((cp / kStages) & 1) ^ 1) || *abort_flag) {
                    *abort_flag = 1;
                    break;
                }
                const int kx = unit_group(u, i, h0, nseg) * g + kc * 64;
                tc::mbar_expect_tx(full(s), kStage);
                tc::tma_load_2d(tileA(s), &mapC, full(s), kx, j0);
#pragma unroll
                for (int t = 0; t < 4; ++t)
                    tc::tma_load_2d(tileB(s, t), &mapT, full(s), kx, t * a.d_pad + m0);
                ++cp;
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------ MMA issuer
        int um = 0;
        for (int i = 0; i < a.G && !*abort_flag; ++i) {
            for (int u = 0; u < nseg; ++u) {
                const int b = um & 1;
                if (!tc::mbar_wait(aempty(b), ((um >> 1) & 1) ^ 1) || *abort_flag) {
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
        }
    } else if (warp >= 2 && warp < kBabaiWarp) {
        // ------------------------------------------------ drain + Babai targets
        const int q = warp & 3, cq = (warp - 2) >> 2;    // lane quarter, 16-column quarter
        const int row = j0 + 32 * q + lane;
        const float *srow = a.S + (size_t)min(row, a.p - 1) * a.G;
        const int dw = warp - 2;
        int ud = 0;
        for (int i = 0; i < a.G; ++i) {
            float hi[16], lo[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                hi[e] = 0.f;
                lo[e] = 0.f;
            }
            bool ok = __all_sync(0xffffffffu, !*abort_flag);
            const int *erow = a.expoT + (size_t)i * a.G;
            int hn = nseg > 0 ? unit_group(0, i, h0, nseg) : 0;
            float s_next = nseg > 0 ? srow[hn] : 0.f;
            int e_next = nseg > 0 ? erow[hn] : 0;
            for (int u = 0; u < nseg && ok; ++u) {
                const int b = ud & 1;
                const float s_cur = row < a.p ? s_next : 0.f;
                const int e_cur = e_next;
                if (u + 1 < nseg) {
                    hn = unit_group(u + 1, i, h0, nseg);
                    s_next = srow[hn];
                    e_next = erow[hn];
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
            // partial of this CTA (slot i & 1: the targets of phase i-1 in
            // every CTA were formed from the other slot before any CTA
            // reaches this point of phase i+1)
            float *th = a.t_hi + (size_t)(i & 1) * a.nks * a.p_pad * g;
            float *tl = a.t_lo + (size_t)(i & 1) * a.nks * a.p_pad * g;
            if (ok && row < a.p) {
                const size_t o = ((size_t)kpart * a.p_pad + row) * g + cpart * 64 + cq * 16;
#pragma unroll
                for (int e = 0; e < 16; e += 4) {
                    float x[4], y[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) two_sum(hi[e + k], lo[e + k], x[k], y[k]);
                    *reinterpret_cast<float4 *>(th + o + e) = make_float4(x[0], x[1], x[2], x[3]);
                    *reinterpret_cast<float4 *>(tl + o + e) = make_float4(y[0], y[1], y[2], y[3]);
                }
            }
            // each thread's partial is visible cluster-wide before the signal
            tc::fence_acq_rel_cluster();
            tc::named_bar_sync(1, 32 * kDrainWarps);
            if (dw == 0 && lane == 0) {
                tc::fence_acq_rel_cluster();
                for (int r = 0; r < kCluster; ++r) tc::count_up_cluster(tc::map_cluster(pcnt, r));
            }
            // the Babai buffers are free once the codes of phase i-1 are out
            bool okw = !*abort_flag;
            if (okw && i >= 1) okw = tc::wait_count_cluster(ccnt, kCluster * i);
            if (okw) okw = tc::wait_count_cluster(pcnt, kCluster * (i + 1));
            okw = __all_sync(0xffffffffu, okw);
            if (!okw) *abort_flag = 1;
            // Babai targets of rows 2 dw, 2 dw + 1 of this CTA's 32:
            // y = (Pt_i - sum of partials) / s in double-float
            if (okw) {
                const int l0 = NT * lane;
#pragma unroll
                for (int rr = 0; rr < 2; ++rr) {
                    const int r = 2 * dw + rr;
                    const int jr = j0 + kRows * rank + r;
                    const int j = min(jr, a.p - 1);
                    const float s = a.S[(size_t)j * a.G + i];
                    const bool live = jr < a.p && a.active[j] != 0 && fabsf(s) > a.eps;
                    const size_t off = (size_t)j * a.d + i * g + l0;
                    float y[NT], yl[NT];
                    if constexpr (NT == 4) {
                        const float4 t0 = *reinterpret_cast<const float4 *>(a.pt_hi + off);
                        const float4 t1 = *reinterpret_cast<const float4 *>(a.pt_lo + off);
                        y[0] = t0.x; y[1] = t0.y; y[2] = t0.z; y[3] = t0.w;
                        yl[0] = t1.x; yl[1] = t1.y; yl[2] = t1.z; yl[3] = t1.w;
                    } else {
                        const float2 t0 = *reinterpret_cast<const float2 *>(a.pt_hi + off);
                        const float2 t1 = *reinterpret_cast<const float2 *>(a.pt_lo + off);
                        y[0] = t0.x; y[1] = t0.y;
                        yl[0] = t1.x; yl[1] = t1.y;
                    }
                    for (int sp = 0; sp < a.nks; ++sp) {
                        const size_t o = ((size_t)sp * a.p_pad + j) * g + l0;
                        float thv[NT], tlv[NT];
                        if constexpr (NT == 4) {
                            const float4 t0 = __ldcg(reinterpret_cast<const float4 *>(th + o));
                            const float4 t1 = __ldcg(reinterpret_cast<const float4 *>(tl + o));
                            thv[0] = t0.x; thv[1] = t0.y; thv[2] = t0.z; thv[3] = t0.w;
                            tlv[0] = t1.x; tlv[1] = t1.y; tlv[2] = t1.z; tlv[3] = t1.w;
                        } else {
                            const float2 t0 = __ldcg(reinterpret_cast<const float2 *>(th + o));
                            const float2 t1 = __ldcg(reinterpret_cast<const float2 *>(tl + o));
                            thv[0] = t0.x; thv[1] = t0.y;
                            tlv[0] = t1.x; tlv[1] = t1.y;
                        }
#pragma unroll
                        for (int t = 0; t < NT; ++t) {
                            const float sm = y[t] - thv[t];
                            const float bb = sm - y[t];
                            const float e = (y[t] - (sm - bb)) + (-thv[t] - bb);
                            y[t] = sm;
                            yl[t] += e - tlv[t];
                        }
                    }
#pragma unroll
                    for (int t = 0; t < NT; ++t) {
                        const float v = live ? (y[t] + yl[t]) / s : 0.f;
                        Yb[uy_idx(l0 + t, r)] = v;
                        Ub[uy_idx(l0 + t, r)] = v;
                    }
                    // codes: one word per 4 coordinates
                    uint32_t packed;
                    if constexpr (NT == 4) {
                        packed = *reinterpret_cast<const uint32_t *>(a.Q + off);
                        Cb[c_idx(lane, r)] = packed;
                    } else {
                        packed = *reinterpret_cast<const uint16_t *>(a.Q + off);
                        const uint32_t other = __shfl_down_sync(0xffffffffu, packed, 1);
                        if ((lane & 1) == 0) Cb[c_idx(lane >> 1, r)] = packed | (other << 16);
                    }
                    if (lane == 0) {
                        rowS[r] = s;
                        rowZ[r] = a.Z[(size_t)j * a.G + i];
                        rowLive[r] = live ? 1 : 0;
                    }
                }
            }
            __threadfence_block();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(ybar);
        }
    } else if (warp == kBabaiWarp) {
        // ------------------------------------------------ Babai, one row per lane
        const int r = lane;
        const int jr = j0 + kRows * rank + r;
        if (lane == 0) {
            tc::mbar_expect_tx(lbar, (uint32_t)(kRpk * sizeof(float)));
            tc::bulk_load(tc::smem_u32(Rs), a.Rpk, kRpk * sizeof(float), lbar);
            ++nl;
        }
        const float qmaxf = (float)a.qmax;
        constexpr float kRound = 12582912.0f;      // 1.5 * 2^23: rounds to nearest even
        for (int i = 0; i < a.G; ++i) {
            bool ok = !*abort_flag && tc::mbar_wait(ybar, i & 1) && tc::mbar_wait(lbar, i & 1);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) {
                *abort_flag = 1;
                break;
            }
            // 1 / R_ll and R_ll of the group
#pragma unroll
            for (int t = 0; t < NT; ++t) {
                const int l = NT * lane + t;
                const float dgv = Rs[rpk_row_off(l, g) + (l & 15)];
                Dg[l] = dgv;
                Rd[l] = 1.0f / dgv;
            }
            __syncwarp();
            const bool live = rowLive[r] != 0;
            const float s = rowS[r];
            // back substitution (Eq. babai_update) relative to the current
            // codes: z + x_l = q_l + u_l / R_ll with u = y - R Delta, blocks of
            // 16 coordinates from the top; the change of the group objective
            // (Eq. group_bils) dF = s^2 sum_l (a_l - y_l)(a_l + y_l),
            // a_l = R_ll Delta_l - u_l, is summed as coordinates become final
            bool any = false;
            float acc = 0.f;
            for (int b0 = g - 16; b0 >= 0; b0 -= 16) {
                float u[16], dq[16];
                uint32_t cw[4];   // current codes of the block, four per word
#pragma unroll
                for (int t = 0; t < 16; ++t) u[t] = Ub[uy_idx(b0 + t, r)];
#pragma unroll
                for (int k = 0; k < 4; ++k) cw[k] = Cb[c_idx((b0 >> 2) + k, r)];
                bool bany = false;
#pragma unroll
                for (int t = 15; t >= 0; --t) {
                    const int l = b0 + t;
                    const float qc = (float)((cw[t >> 2] >> (8 * (t & 3))) & 0xFFu);
                    const float x = fmaf(u[t], Rd[l], qc);
                    const float qv =
                        fminf(fmaxf(__fsub_rn(__fadd_rn(x, kRound), kRound), 0.f), qmaxf);
                    dq[t] = live ? qv - qc : 0.f;
                    bany |= dq[t] != 0.f;
#pragma unroll
                    for (int tt = 0; tt < t; ++tt)
                        u[tt] = fmaf(-Rs[rpk_row_off(b0 + tt, g) + t], dq[t], u[tt]);
                    // coordinate l is final
                    const float av = Dg[l] * dq[t] - u[t];
                    const float yv = Yb[uy_idx(l, r)];
                    acc = fmaf(av - yv, av + yv, acc);
                }
                any |= bany;
                // proposed codes of the block (current code + integer change)
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    uint32_t w = 0;
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int c = (int)((cw[k] >> (8 * e)) & 0xFFu) + (int)dq[4 * k + e];
                        w |= (uint32_t)c << (8 * e);
                    }
                    Cb[c_idx((b0 >> 2) + k, r)] = w;
                }
                // column updates of the coordinates below the block, in
                // descending column order
                if (__any_sync(0xffffffffu, bany)) {
#pragma unroll 2
                    for (int l = 0; l < b0; ++l) {
                        const float4 *rr = reinterpret_cast<const float4 *>(
                            Rs + rpk_row_off(l, g) + (b0 - 16 * (l >> 4)));
                        float rv[16];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const float4 v4 = rr[k];
                            rv[4 * k] = v4.x; rv[4 * k + 1] = v4.y;
                            rv[4 * k + 2] = v4.z; rv[4 * k + 3] = v4.w;
                        }
                        float ul = Ub[uy_idx(l, r)];
#pragma unroll
                        for (int t = 15; t >= 0; --t) ul = fmaf(-rv[t], dq[t], ul);
                        Ub[uy_idx(l, r)] = ul;
                    }
                }
            }
            const float dF = s * s * acc;
            const bool accept = live && any && isfinite(dF) && dF < 0.f;
            if (accept) {
                const int j = jr;
                const int z = rowZ[r];
                const size_t off = (size_t)j * a.d + i * g;
                __half *crow = a.cplane + (size_t)j * a.d_pad + i * g;
#pragma unroll 2
                for (int k4 = 0; k4 < g / 16; ++k4) {
                    uint32_t w[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) w[k] = Cb[c_idx(4 * k4 + k, r)];
                    *reinterpret_cast<uint4 *>(a.Q + off + 16 * k4) = make_uint4(w[0], w[1], w[2], w[3]);
                    uint32_t hw[8];
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        const uint32_t c0 = (w[k >> 1] >> (16 * (k & 1))) & 0xFFu;
                        const uint32_t c1 = (w[k >> 1] >> (16 * (k & 1) + 8)) & 0xFFu;
                        const __half h0v = __int2half_rn((int)c0 - z);
                        const __half h1v = __int2half_rn((int)c1 - z);
                        hw[k] = (uint32_t)__half_as_ushort(h0v) | ((uint32_t)__half_as_ushort(h1v) << 16);
                    }
                    uint4 *cdst = reinterpret_cast<uint4 *>(crow + 16 * k4);
                    cdst[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
                    cdst[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
                }
                a.accepted[j] += 1;
            }
            // the accepted codes reach the other CTAs' tensor-map loads
            tc::fence_proxy_async_global();
            tc::fence_acq_rel_cluster();
            __syncwarp();
            if (lane == 0) {
                if (i + 1 < a.G) {
                    // the next group's factor (this phase is done with the buffer)
                    tc::fence_proxy_async_smem();
                    tc::mbar_expect_tx(lbar, (uint32_t)(kRpk * sizeof(float)));
                    tc::bulk_load(tc::smem_u32(Rs), a.Rpk + (size_t)(i + 1) * kRpk,
                                  kRpk * sizeof(float), lbar);
                    ++nl;
                }
                tc::fence_acq_rel_cluster();
                for (int rk = 0; rk < kCluster; ++rk) tc::count_up_cluster(tc::map_cluster(ccnt, rk));
            }
            __syncwarp();
        }
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
    }
    if (warp == kBabaiWarp && lane == 0 && nl > 0) {
        if (!tc::mbar_wait(lbar, (nl - 1) & 1)) *abort_flag = 1;
    }
    tc::tc_fence_before();
    __syncwarp();
    // no CTA leaves while another may still arrive on its barriers
    tc::cluster_sync();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, ST_TIMEOUT);
}

}  // namespace

int sweep_k_parts(int g) { return kCluster / (g / 64); }

int sweep_rpk_size(int g) { return rpk_size(g); }

// R_i in the packed row layout of the sweep kernel, from L_i = R_i^T
// (row-major); entries left of the diagonal are zero.
__global__ void pack_rfactor_kernel(const float *__restrict__ Lf, float *__restrict__ Rpk, int g) {
    const int i = blockIdx.x;
    const float *L = Lf + (size_t)i * g * g;
    float *out = Rpk + (size_t)i * rpk_size(g);
    for (int l = threadIdx.y; l < g; l += blockDim.y) {
        const int c0 = 16 * (l >> 4);
        for (int h = c0 + threadIdx.x; h < g; h += blockDim.x)
            out[rpk_row_off(l, g) + (h - c0)] = h >= l ? L[(size_t)h * g + l] : 0.f;
    }
}

cudaError_t launch_pack_rfactor(const float *Lf, float *Rpk, int G, int g, cudaStream_t s) {
    pack_rfactor_kernel<<<G, dim3(32, 8), 0, s>>>(Lf, Rpk, g);
    return cudaGetLastError();
}

cudaError_t launch_sweep(const CUtensorMap &mapC, const CUtensorMap &mapT, float *t_hi,
                         float *t_lo, const float *pt_hi, const float *pt_lo, const float *Rpk,
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
    SweepArgs a{t_hi, t_lo, pt_hi, pt_lo, Rpk, S, expoT, Q, Z, cplane, active, accepted, status,
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
