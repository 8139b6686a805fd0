// Target projection P = W H on the tensor cores, exact to double-float
// accuracy, and the quantities derived from it.  For the main target the
// reduced target is R W, so the right-hand side of Eq.
// scale_normal_equations is rhs_j[i] = c_i^T P_j[grp i] with P_j = H w_j
// (App. G "Computational Complexity", the target-projection shortcut), and
// the objective is F_j = w_j^T H w_j - 2 s^T rhs_j + s^T Gram_j s.
//
// Both operands are written in integer digits so that every tensor-core
// partial sum is exact:
//   W[j, k] = 2^(ew(j,h) - 7) sum_{t<4} a_t 2^(-8t),  k in group h, one exponent
//             per (row, group) with max |W[j, grp h]| <= 2^ew;
//   H[k, m] = 2^(E(h,n) - 7) sum_{u<6} b_u 2^(-8u),   the block exponent of
//             block (h, n), n = the group of m,
// with |a_t|, |b_u| <= 128 (exact in bf16).  Four digits hold every float32 W
// entry within 2^7 of its group maximum exactly, six every H entry within
// 2^24 of its block maximum.  For each group h of K the eighteen digit
// products with t + u <= 5 (six MMAs per K step) accumulate in six TMEM
// "levels" l = t + u; a level sums at most 4 x 128 products of 14-bit
// integers per output, an exact integer below 2^23.  The epilogue combines the levels in
// double-float (pairs of float32), applies 2^(ew + E - 14) and adds the
// group's contribution to a double-float accumulator.  The dropped products
// (t + u >= 6) are below 2^-48 of the block scales.
//
// Roles: warp 0 TMA producer (4 W planes + 6 H planes per 64-wide K chunk),
// warp 1 TMEM allocation and MMA issue, warps 2..9 drain (warp w reads TMEM
// lanes 32 (w % 4) and 32 of the tile's 64 columns).  Tile 128 x 64; the six
// levels take 384 TMEM columns, single-buffered: the drain warps release
// them as soon as their loads have landed and combine from registers while
// the next group's products run.
#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kWDig = 4, kHDig = 6, kLevels = 6;
constexpr int kTileA = 128 * 64 * 2;   // one W digit plane, 128 rows x 64 K
constexpr int kTileB = 64 * 64 * 2;    // one H digit plane, 64 rows x 64 K
// WDIG row-side digit planes (4 for W, 6 for the double-float P of the folded
// projection); DIAG: only the K block of the tile's own column group (the
// block-diagonal right-hand side R_i^{-1}), one stage of 144 KB.
template <int WDIG, bool DIAG>
struct ProjCfg {
    static constexpr int kStage = WDIG * kTileA + kHDig * kTileB;
    static constexpr int kStages = DIAG ? 1 : 2;
    static constexpr int kSmem = 1024 + kStages * kStage + 256;
};
// For a W digit t the H digit planes u are consecutive 64-row tiles and the
// levels t + u consecutive 64-column blocks, so one MMA covers up to four
// planes (N = 64 per plane).
__host__ __device__ constexpr uint32_t idesc_n(int n) { return tc::idesc_bf16_f32(128, n); }
constexpr int kGroupRows = 8;

struct ProjArgs {
    float *Phi, *Plo;    // [p][d] double-float result
    const int *wexp;     // [p][G] row-group exponents of W
    const int *hexp;     // [G][G] block exponents of H ([G] in the diagonal form)
    int *status;
    int p, d, g, G, w_plane, h_plane;   // rows between digit planes in the two maps
};

// (s, e) with s + e = a + b exactly
__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

template <int WDIG, bool DIAG>
__global__ void __launch_bounds__(320, 1)
    tc_proj_kernel(const __grid_constant__ CUtensorMap mapW, const __grid_constant__ CUtensorMap mapH,
                   ProjArgs a) {
    constexpr int kStage = ProjCfg<WDIG, DIAG>::kStage, kStages = ProjCfg<WDIG, DIAG>::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *bars = (uint64_t *)(smem + kStages * kStage);
    uint32_t *tmem_slot = (uint32_t *)(bars + 2 * kStages + 2);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nkc = a.g / 64;               // K chunks per group
    // General form: one 128 x 64 tile per CTA in grouped order (bands of
    // kGroupRows row tiles sweep all column tiles), one segment per group of
    // K.  Diagonal form: the CTA loops over tiles, item blockIdx.x + v gridDim.x
    // of (row tiles) x (d / 64 column tiles), one segment each: the K block of
    // the tile's own column group.
    int gj0 = 0, gn0 = 0;
    if (!DIAG) {
        const int lin = blockIdx.y * gridDim.x + blockIdx.x;
        const int per_band = kGroupRows * gridDim.y;
        const int band = lin / per_band, in_band = lin % per_band;
        const int rows_in_band = min(kGroupRows, (int)gridDim.x - band * kGroupRows);
        gj0 = (band * kGroupRows + in_band % rows_in_band) * 128;
        gn0 = (in_band / rows_in_band) * 64;
    }
    const int nct = a.d / 64;
    const int nitems = DIAG ? ((a.p + 127) / 128) * nct : 1;
    const int nseg = DIAG ? ((int)blockIdx.x < nitems ? (nitems - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0)
                          : a.G;
    const int nchunks = nseg * nkc;
    // tile (first row, first column) of segment v; a 64-wide tile lies in
    // one column group n0 / g
    auto tile_of = [&](int v, int &j0, int &n0) {
        if (DIAG) {
            const int it = (int)blockIdx.x + v * (int)gridDim.x;
            j0 = (it / nct) * 128;
            n0 = (it % nct) * 64;
        } else {
            j0 = gj0;
            n0 = gn0;
        }
    };

    auto full = [&](int s) { return tc::smem_u32(bars + s); };
    auto empty = [&](int s) { return tc::smem_u32(bars + kStages + s); };
    const uint32_t afull = tc::smem_u32(bars + 2 * kStages);
    const uint32_t aempty = tc::smem_u32(bars + 2 * kStages + 1);
    auto tileA = [&](int s, int t) { return tc::smem_u32(smem + s * kStage + t * kTileA); };
    auto tileB = [&](int s, int u) {
        return tc::smem_u32(smem + s * kStage + WDIG * kTileA + u * kTileB);
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(full(s), 1);
            tc::mbar_init(empty(s), 1);
        }
        tc::mbar_init(afull, 1);
        tc::mbar_init(aempty, 8);
        *abort_flag = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(tc::smem_u32(tmem_slot), 512);
        tc::tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tc::prefetch_tmap(&mapW);
        tc::prefetch_tmap(&mapH);
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0 && lane == 0) {
        // ---------------- producer
        int issued = 0;
        for (int c = 0; c < nchunks; ++c) {
            const int s = c % kStages;
            if (!tc::mbar_wait(empty(s), ((c / kStages) & 1) ^ 1) || *abort_flag) {
                *abort_flag = 1;
                break;
            }
            const int v = c / nkc, kc = c % nkc;
            int j0, n0;
            tile_of(v, j0, n0);
            // K offsets in the two maps: the right-hand side of the diagonal
            // form holds only the g columns of each group's block
            const int kw = DIAG ? (n0 / a.g) * a.g + kc * 64 : c * 64;
            const int kh = DIAG ? kc * 64 : c * 64;
            tc::mbar_expect_tx(full(s), kStage);
#pragma unroll
            for (int t = 0; t < WDIG; ++t)
                tc::tma_load_2d(tileA(s, t), &mapW, full(s), kw, t * a.w_plane + j0);
#pragma unroll
            for (int u = 0; u < kHDig; ++u)
                tc::tma_load_2d(tileB(s, u), &mapH, full(s), kh, u * a.h_plane + n0);
            issued = c + 1;
        }
        // do not leave with copies in flight
        for (int c = issued > kStages ? issued - kStages : 0; c < issued; ++c)
            if (!tc::mbar_wait(full(c % kStages), (c / kStages) & 1)) *abort_flag = 1;
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        for (int sg = 0; sg < nseg && !*abort_flag; ++sg) {
            if (!tc::mbar_wait(aempty, (sg & 1) ^ 1)) {
                *abort_flag = 1;
                break;
            }
            tc::tc_fence_after();
            for (int kc = 0; kc < nkc; ++kc) {
                const int c = sg * nkc + kc;
                const int s = c % kStages;
                if (!tc::mbar_wait(full(s), (c / kStages) & 1) || *abort_flag) {
                    *abort_flag = 1;
                    break;
                }
                tc::tc_fence_after();
#pragma unroll
                for (int sub = 0; sub < 4; ++sub) {
#pragma unroll
                    for (int t = 0; t < WDIG; ++t) {
                        const uint64_t ad = tc::sdesc_sw128(tileA(s, t)) + 2 * sub;
                        // the products of W digit t with H digits u < kLevels - t,
                        // in runs of at most four planes; t = 0 opens every level
                        const uint32_t acc = (kc | sub | t) != 0;
#pragma unroll
                        for (int u0 = 0; u0 < kLevels - t; u0 += 4) {
                            const int nu = min(4, kLevels - t - u0);
                            const uint64_t bd = tc::sdesc_sw128(tileB(s, u0)) + 2 * sub;
                            tc::mma_bf16(tmem + (t + u0) * 64, ad, bd, idesc_n(64 * nu), acc);
                        }
                    }
                }
                tc::mma_commit(empty(s));
            }
            tc::mma_commit(afull);
        }
    } else if (warp >= 2) {
        // ---------------- drain: levels -> double-float per group -> accumulator
        if constexpr (DIAG) {
            // diagonal form: a tile per segment, written when it completes
            const int q = warp & 3, half = (warp - 2) >> 2;
            float hi[32], lo[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                hi[e] = 0.f;
                lo[e] = 0.f;
            }
            bool ok = true;
            const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + half * 32;
            // exponents of this thread's row and segment v: W's (row, K group)
            // and H's block (K group, column group); loaded one segment ahead
            auto seg_exp = [&](int v, int &ew, int &eh) {
                int j0, n0;
                tile_of(v, j0, n0);
                const int row = j0 + 32 * q + lane, hb = n0 / a.g, kg = DIAG ? hb : v;
                ew = row < a.p ? a.wexp[(size_t)row * a.G + kg] : 0;
                eh = hb < a.G ? a.hexp[DIAG ? hb : kg * a.G + hb] : 0;
            };
            int ew_next = 0, eh_next = 0;
            if (nseg > 0) seg_exp(0, ew_next, eh_next);
            for (int sg = 0; sg < nseg; ++sg) {
                const int ew = ew_next, eh = eh_next;
                if (sg + 1 < nseg) seg_exp(sg + 1, ew_next, eh_next);
                bool w = tc::mbar_wait(afull, sg & 1);
                w = __shfl_sync(0xffffffffu, w && !*abort_flag, 0);
                tc::tc_fence_after();
                if (!w) {
                    ok = false;
                    *abort_flag = 1;
                    break;
                }
                const float scale = ldexpf(1.0f, ew + eh - 14);
                // value of the group = sum_l L_l 2^(-8 l), as (vh, vl), 32 columns
                float vh[32], vl[32];
#pragma unroll
                for (int l = 0; l < kLevels; ++l) {
                    uint32_t x[32];
                    tc::tmem_ld32(base + l * 64, x);
                    tc::tmem_wait_ld();
                    if (l == kLevels - 1) {
                        // every level is in registers: hand the columns back
                        tc::tc_fence_before();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(aempty);
                    }
                    const float f = ldexpf(1.0f, -8 * l);
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        const float v = __uint_as_float(x[e]) * f;   // exact (power of two)
                        if (l == 0) {
                            vh[e] = v;
                            vl[e] = 0.f;
                        } else {
                            float s2, e2;
                            two_sum(vh[e], v, s2, e2);
                            vh[e] = s2;
                            vl[e] += e2;
                        }
                    }
                }
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    float s2, e2;
                    two_sum(hi[e], vh[e] * scale, s2, e2);
                    hi[e] = s2;
                    lo[e] += e2 + vl[e] * scale;
                }
                // the tile is complete after its last segment (every segment in
                // the diagonal form)
                if (DIAG || sg + 1 == nseg) {
                    int j0, n0;
                    tile_of(sg, j0, n0);
                    const int row = j0 + 32 * q + lane, ncol = n0 + half * 32;
                    if (row < a.p) {
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            const int col = ncol + e;
                            if (col < a.d) {
                                float s2, e2;
                                two_sum(hi[e], lo[e], s2, e2);
                                a.Phi[(size_t)row * a.d + col] = s2;
                                a.Plo[(size_t)row * a.d + col] = e2;
                            }
                        }
                    }
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        hi[e] = 0.f;
                        lo[e] = 0.f;
                    }
                }
            }
            (void)ok;
        } else {
            const int q = warp & 3, half = (warp - 2) >> 2;
            const int j0 = gj0, n0 = gn0, hblk = n0 / a.g;
            const int row = j0 + 32 * q + lane;
            float hi[32], lo[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                hi[e] = 0.f;
                lo[e] = 0.f;
            }
            bool ok = true;
            const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + half * 32;
            // exponents of the next group, loaded one group ahead
            const int *wrow = a.wexp + (size_t)min(row, a.p - 1) * a.G;
            const int hb = min(hblk, a.G - 1);
            int ew_next = wrow[0], eh_next = a.hexp[hb];
            for (int sg = 0; sg < nseg; ++sg) {
                const int ew = row < a.p ? ew_next : 0;
                const int eh = hblk < a.G ? eh_next : 0;
                if (sg + 1 < nseg) {
                    ew_next = wrow[sg + 1];
                    eh_next = a.hexp[(sg + 1) * a.G + hb];
                }
                bool w = tc::mbar_wait(afull, sg & 1);
                w = __shfl_sync(0xffffffffu, w && !*abort_flag, 0);
                tc::tc_fence_after();
                if (!w) {
                    ok = false;
                    *abort_flag = 1;
                    break;
                }
                const float scale = ldexpf(1.0f, ew + eh - 14);
                // value of the group = sum_l L_l 2^(-8 l), as (vh, vl), 32 columns
                float vh[32], vl[32];
#pragma unroll
                for (int l = 0; l < kLevels; ++l) {
                    uint32_t x[32];
                    tc::tmem_ld32(base + l * 64, x);
                    tc::tmem_wait_ld();
                    if (l == kLevels - 1) {
                        // every level is in registers: hand the columns back
                        tc::tc_fence_before();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(aempty);
                    }
                    const float f = ldexpf(1.0f, -8 * l);
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        const float v = __uint_as_float(x[e]) * f;   // exact (power of two)
                        if (l == 0) {
                            vh[e] = v;
                            vl[e] = 0.f;
                        } else {
                            float s2, e2;
                            two_sum(vh[e], v, s2, e2);
                            vh[e] = s2;
                            vl[e] += e2;
                        }
                    }
                }
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    float s2, e2;
                    two_sum(hi[e], vh[e] * scale, s2, e2);
                    hi[e] = s2;
                    lo[e] += e2 + vl[e] * scale;
                }
            }
            if (ok && row < a.p) {
                const int ncol = n0 + half * 32;
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const int col = ncol + e;
                    if (col < a.d) {
                        float s2, e2;
                        two_sum(hi[e], lo[e], s2, e2);
                        a.Phi[(size_t)row * a.d + col] = s2;
                        a.Plo[(size_t)row * a.d + col] = e2;
                    }
                }
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, ST_TIMEOUT);
}

// Digits of W per (row, group): x = W 2^(7 - ew) in [-128, 128] with
// max |W[j, grp h]| <= 2^ew; a_0 = rint(x), a_t = rint(256 * remainder).
// One warp per (row, group).
__global__ void slice_rows_kernel(const float *__restrict__ W, __nv_bfloat16 *__restrict__ planes,
                                  int *__restrict__ wexp, int p, int d, int d_pad, int p_pad, int g) {
    const int G = d / g;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (warp >= (long long)p * G) return;
    const int j = (int)(warp / G), h = (int)(warp % G);
    const float *src = W + (size_t)j * d + (size_t)h * g;
    float mx = 0.f;
    for (int m = lane; m < g; m += 32) mx = fmaxf(mx, fabsf(src[m]));
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    int e = 0;
    if (mx > 0.f) frexpf(mx, &e);
    if (lane == 0) wexp[(size_t)j * G + h] = e;
    const size_t plane = (size_t)p_pad * d_pad;
    for (int m = lane; m < g; m += 32) {
        float x = ldexpf(src[m], 7 - e);
        const size_t off = (size_t)j * d_pad + (size_t)h * g + m;
#pragma unroll
        for (int t = 0; t < kWDig; ++t) {
            const float dg = rintf(x);
            planes[t * plane + off] = __float2bfloat16_rn(dg);
            x = (x - dg) * 256.f;
        }
    }
}

// Exact product c * (ph + pl) added to the double-float (sh, sl): c is a small
// integer, so c * ph splits exactly by one fma.
__device__ __forceinline__ void df_axpy(float c, float ph, float pl, float &sh, float &sl) {
    const float m = c * ph;
    const float me = fmaf(c, ph, -m);
    float s2, e2;
    two_sum(sh, m, s2, e2);
    sh = s2;
    sl += e2 + fmaf(c, pl, me);
}

__device__ __forceinline__ void df_warp_sum(float &sh, float &sl) {
    for (int o = 16; o; o >>= 1) {
        const float oh = __shfl_xor_sync(0xffffffffu, sh, o);
        const float ol = __shfl_xor_sync(0xffffffffu, sl, o);
        float s2, e2;
        two_sum(sh, oh, s2, e2);
        sh = s2;
        sl += e2 + ol;
    }
}

// rhs_j[i] = sum_{l in grp i} (q_l - z_i) P_j[l], one warp per row, lane owns
// NT = g/32 consecutive entries of every group.
template <int NT>
__global__ void rhs_kernel(const uint8_t *__restrict__ Q, const int32_t *__restrict__ Z,
                           const float *__restrict__ Phi, const float *__restrict__ Plo,
                           const int *__restrict__ active, double *__restrict__ rhs, int p, int d) {
    constexpr int g = 32 * NT;
    const int G = d / g;
    const int j = (int)(((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (j >= p || (active && !active[j])) return;   // warp-uniform
    const size_t off = (size_t)j * d + NT * lane;
    for (int i = 0; i < G; ++i) {
        const float z = (float)Z[(size_t)j * G + i];
        const size_t o = off + (size_t)i * g;
        float ph[NT], pl[NT], qc[NT];
        if constexpr (NT == 4) {
            const float4 a4 = *reinterpret_cast<const float4 *>(Phi + o);
            const float4 b4 = *reinterpret_cast<const float4 *>(Plo + o);
            const uint32_t q4 = *reinterpret_cast<const uint32_t *>(Q + o);
            ph[0] = a4.x; ph[1] = a4.y; ph[2] = a4.z; ph[3] = a4.w;
            pl[0] = b4.x; pl[1] = b4.y; pl[2] = b4.z; pl[3] = b4.w;
#pragma unroll
            for (int t = 0; t < 4; ++t) qc[t] = (float)((q4 >> (8 * t)) & 0xFFu);
        } else {
            const float2 a2 = *reinterpret_cast<const float2 *>(Phi + o);
            const float2 b2 = *reinterpret_cast<const float2 *>(Plo + o);
            const uint32_t q2 = *reinterpret_cast<const uint16_t *>(Q + o);
            ph[0] = a2.x; ph[1] = a2.y;
            pl[0] = b2.x; pl[1] = b2.y;
            qc[0] = (float)(q2 & 0xFFu);
            qc[1] = (float)(q2 >> 8);
        }
        float sh = 0.f, sl = 0.f;
#pragma unroll
        for (int t = 0; t < NT; ++t) df_axpy(qc[t] - z, ph[t], pl[t], sh, sl);
        df_warp_sum(sh, sl);
        if (lane == 0) rhs[(size_t)j * G + i] = (double)sh + (double)sl;
    }
}

// wHw_j = sum_k W[j,k] P[j,k] with P = Phi + Plo, double-float per lane, one
// warp per row.
__global__ void whw_kernel(const float *__restrict__ W, const float *__restrict__ Phi,
                           const float *__restrict__ Plo, double *__restrict__ out, int p, int d) {
    const int j = (int)(((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (j >= p) return;
    const size_t off = (size_t)j * d;
    float sh = 0.f, sl = 0.f;
    for (int k = lane; k < d; k += 32) {
        const float w = W[off + k], ph = Phi[off + k], pl = Plo[off + k];
        const float m = w * ph;
        const float me = fmaf(w, ph, -m);
        float s2, e2;
        two_sum(sh, m, s2, e2);
        sh = s2;
        sl += e2 + fmaf(w, pl, me);
    }
    df_warp_sum(sh, sl);
    if (lane == 0) out[j] = (double)sh + (double)sl;
}

// Propagation-corrected target (App. "Propagation-Corrected Targets and
// QEP", Eqs. mu-target, w-corr).  With H = X~^T X~ + nu^2 I and K = X~^T X,
// the projection of the corrected weights needs no inverse of H:
//   H w_corr = A^T y(mu) = mu H w + (1 - mu) (K w + nu^2 w),
// and the target energy that replaces w^T H w in the objective is
//   ||y(mu)||^2 = (1-mu)^2 w^T XX w + 2 mu (1-mu) w^T K w
//                 + mu^2 (w^T H w - nu^2 w^T w) + nu^2 w^T w.
// On entry P = Phi + Plo holds H w, PK = Khi + Klo holds K w (rows of the
// target projection with K in place of H), wHw[j] = w^T H w and
// wXXw[j] = w^T XX w; on exit P holds H w_corr and wHw[j] ||y_j(mu)||^2.
// One warp per row, float64 arithmetic.
__global__ void mu_combine_kernel(float *__restrict__ Phi, float *__restrict__ Plo,
                                  const float *__restrict__ Khi, const float *__restrict__ Klo,
                                  const float *__restrict__ W, const double *__restrict__ wXXw,
                                  double *__restrict__ wHw, int p, int d, double mu, double nu2) {
    const int j = (int)(((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    const int lane = threadIdx.x & 31;
    if (j >= p) return;
    const size_t off = (size_t)j * d;
    double wKw = 0.0, ww = 0.0;
    for (int k = lane; k < d; k += 32) {
        const double P = (double)Phi[off + k] + (double)Plo[off + k];
        const double PK = (double)Khi[off + k] + (double)Klo[off + k];
        const double w = W[off + k];
        const double r = mu * P + (1.0 - mu) * fma(nu2, w, PK);
        const float hi = __double2float_rn(r);
        Phi[off + k] = hi;
        Plo[off + k] = __double2float_rn(r - (double)hi);
        wKw = fma(w, PK, wKw);
        ww = fma(w, w, ww);
    }
    for (int o = 16; o; o >>= 1) {
        wKw += __shfl_xor_sync(0xffffffffu, wKw, o);
        ww += __shfl_xor_sync(0xffffffffu, ww, o);
    }
    if (lane == 0) {
        const double a = 1.0 - mu;
        wHw[j] = a * a * wXXw[j] + 2.0 * mu * a * wKw + mu * mu * (wHw[j] - nu2 * ww) + nu2 * ww;
    }
}

// Digits of the double-float P for the folded projection: per (row, group)
// the exponent e with max |P| < 2^e, and six balanced base-256 digits of
// P 2^(7-e) (|digit| <= 128, exact in bf16), taken from the float pair
// (xh, xl) = (Phi, Plo) 2^(7-e) with exact float operations: the digit is
// rint(xh), and the remainder (xh - digit) + xl is renormalised by an exact
// two-sum before the next digit.  Six digits hold P to 2^-48 of its group
// maximum (the pair itself carries about 48 bits).
__global__ void slice_df_rows_kernel(const float *__restrict__ Phi, const float *__restrict__ Plo,
                                     __nv_bfloat16 *__restrict__ planes, int *__restrict__ pexp,
                                     int p, int d, int d_pad, int p_pad, int g) {
    const int G = d / g;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (warp >= (long long)p * G) return;
    const int j = (int)(warp / G), h = (int)(warp % G);
    const size_t src = (size_t)j * d + (size_t)h * g;
    float mx = 0.f;
    for (int m = lane; m < g; m += 32) mx = fmaxf(mx, fabsf(Phi[src + m]));
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    int e = 0;
    if (mx > 0.f) frexpf(mx, &e);
    if (lane == 0) pexp[(size_t)j * G + h] = e;
    const size_t plane = (size_t)p_pad * d_pad;
    for (int m = lane; m < g; m += 32) {
        float xh = ldexpf(Phi[src + m], 7 - e), xl = ldexpf(Plo[src + m], 7 - e);
        const size_t off = (size_t)j * d_pad + (size_t)h * g + m;
#pragma unroll
        for (int t = 0; t < kHDig; ++t) {
            const float dg = rintf(xh);
            planes[t * plane + off] = __float2bfloat16_rn(dg);
            float s2, e2;
            two_sum(xh - dg, xl, s2, e2);
            xh = s2 * 256.f;
            xl = e2 * 256.f;
        }
    }
}

// Digits of the group inverses for the folded projection (once per prepared
// Hessian): plane u, row i g + a, column b holds digit u of R_i^{-1}[b][a]
// (zero below the diagonal), so that the 64 x 64 tiles of the projection
// kernel read the transposed block; exponent E_i with max |R_i^{-1}| < 2^E_i,
// six balanced base-256 digits of R_i^{-1} 2^(7-E_i) in float64.
__global__ void slice_rinv_kernel(const double *__restrict__ Rinv, __nv_bfloat16 *__restrict__ rdig,
                                  int *__restrict__ rexp, int d, int g) {
    __shared__ double red[32];
    const int i = blockIdx.x;
    const double *Ri = Rinv + (size_t)i * g * g;
    double mx = 0.0;
    for (int idx = threadIdx.x; idx < g * g; idx += blockDim.x) mx = fmax(mx, fabs(Ri[idx]));
    for (int o = 16; o; o >>= 1) mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
    __syncthreads();
    if (threadIdx.x < 32) {
        mx = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.0;
        for (int o = 16; o; o >>= 1) mx = fmax(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if (threadIdx.x == 0) red[0] = mx;
    }
    __syncthreads();
    mx = red[0];
    int E = 0;
    if (mx > 0.0) frexp(mx, &E);
    if (threadIdx.x == 0) rexp[i] = E;
    const size_t plane = (size_t)d * g;
    for (int idx = threadIdx.x; idx < g * g; idx += blockDim.x) {
        const int a = idx / g, b = idx % g;
        double x = b <= a ? ldexp(Ri[(size_t)b * g + a], 7 - E) : 0.0;
        const size_t off = ((size_t)i * g + a) * g + b;
#pragma unroll
        for (int u = 0; u < kHDig; ++u) {
            const double dg = rint(x);
            rdig[u * plane + off] = __float2bfloat16_rn((float)dg);
            x = (x - dg) * 256.0;
        }
    }
}

}  // namespace

cudaError_t launch_slice_rinv(const double *Rinv, __nv_bfloat16 *rdig, int *rexp, int d, int g,
                              cudaStream_t s) {
    slice_rinv_kernel<<<d / g, 256, 0, s>>>(Rinv, rdig, rexp, d, g);
    return cudaGetLastError();
}

// Pt = the folded projection, Pt[j, i g + a] = sum_{b <= a} R_i^{-1}[b][a] P[j, i g + b]:
// the six digit planes of P (into the row-digit workspace) and the
// block-diagonal product with the digits of R_i^{-1} on the tensor cores.
cudaError_t launch_ptilde(const CUtensorMap &mapPd, const CUtensorMap &mapR, const float *Phi,
                          const float *Plo, __nv_bfloat16 *pdig, int *pexp, const int *rexp,
                          float *out_hi, float *out_lo, int p, int p_pad, int d, int d_pad, int g,
                          int *status, cudaStream_t s) {
    const long long warps = (long long)p * (d / g);
    slice_df_rows_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, s>>>(
        Phi, Plo, pdig, pexp, p, d, d_pad, p_pad, g);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    using C = ProjCfg<kHDig, true>;
    static std::atomic<unsigned long long> attr_done{0};
    e = set_max_dynamic_smem((const void *)tc_proj_kernel<kHDig, true>, C::kSmem, attr_done);
    if (e != cudaSuccess) return e;
    ProjArgs a{out_hi, out_lo, pexp, rexp, status, p, d, g, d / g, p_pad, d};
    // persistent: one CTA per SM over the (p_pad / 128) x (d / 64) tiles
    (void)d_pad;
    const int items = (p_pad / 128) * (d / 64);
    const int ctas = items < num_sms() ? items : num_sms();
    tc_proj_kernel<kHDig, true><<<dim3(ctas, 1, 1), 320, C::kSmem, s>>>(mapPd, mapR, a);
    return cudaGetLastError();
}

cudaError_t launch_slice_rows(const float *W, __nv_bfloat16 *planes, int *wexp, int p, int d,
                              int d_pad, int p_pad, int g, cudaStream_t s) {
    const long long warps = (long long)p * (d / g);
    slice_rows_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, s>>>(W, planes, wexp, p, d,
                                                                          d_pad, p_pad, g);
    return cudaGetLastError();
}

cudaError_t launch_tc_proj(const CUtensorMap &mapW, const CUtensorMap &mapH, float *Phi,
                           float *Plo, const int *wexp, const int *hexp, int p, int p_pad, int d,
                           int d_pad, int g, int *status, cudaStream_t s) {
    using C = ProjCfg<kWDig, false>;
    static std::atomic<unsigned long long> attr_done{0};
    const cudaError_t e =
        set_max_dynamic_smem((const void *)tc_proj_kernel<kWDig, false>, C::kSmem, attr_done);
    if (e != cudaSuccess) return e;
    ProjArgs a{Phi, Plo, wexp, hexp, status, p, d, g, d / g, p_pad, d_pad};
    dim3 grid(p_pad / 128, d_pad / 64, 1);
    tc_proj_kernel<kWDig, false><<<grid, 320, C::kSmem, s>>>(mapW, mapH, a);
    return cudaGetLastError();
}

cudaError_t launch_whw(const float *W, const float *Phi, const float *Plo, double *out, int p,
                       int d, cudaStream_t s) {
    whw_kernel<<<(unsigned)(((long long)p * 32 + 255) / 256), 256, 0, s>>>(W, Phi, Plo, out, p, d);
    return cudaGetLastError();
}

cudaError_t launch_mu_combine(float *Phi, float *Plo, const float *Khi, const float *Klo,
                              const float *W, const double *wXXw, double *wHw, int p, int d,
                              double mu, double nu2, cudaStream_t s) {
    mu_combine_kernel<<<(unsigned)(((long long)p * 32 + 255) / 256), 256, 0, s>>>(
        Phi, Plo, Khi, Klo, W, wXXw, wHw, p, d, mu, nu2);
    return cudaGetLastError();
}

cudaError_t launch_rhs(const uint8_t *Q, const int32_t *Z, const float *Phi, const float *Plo,
                       const int *active, double *rhs, int p, int d, int g, cudaStream_t s) {
    const unsigned blocks = (unsigned)(((long long)p * 32 + 255) / 256);
    if (g == 128)
        rhs_kernel<4><<<blocks, 256, 0, s>>>(Q, Z, Phi, Plo, active, rhs, p, d);
    else if (g == 64)
        rhs_kernel<2><<<blocks, 256, 0, s>>>(Q, Z, Phi, Plo, active, rhs, p, d);
    else
        return cudaErrorInvalidValue;
    return cudaGetLastError();
}

}  // namespace jarq
