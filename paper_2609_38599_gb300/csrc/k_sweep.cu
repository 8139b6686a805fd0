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
// global memory.  Each CTA then runs the Babai proposals of its 32 rows of
// the tile on the targets
//     y = (Pt_i - T_i) / s_i = R_i^{-T} (H r)_i / s_i
// formed from the partials of all four CTAs.
//
// Overlap.  Group i's codes change only in phase i, so the product of phase
// i+1 needs phase i's result only for the K chunks of group i.  The CTA
// whose K range holds group i takes that group last in phase i+1, and its
// producer waits for the codes of all four CTAs only before loading it.
// The Babai proposals of phase i therefore run on their own warps while the
// product of phase i+1 streams through the tensor cores: the product is
// bound by the tile loads of each SM, and the drain warps that combine its
// digit sums are idle most of the time, so a phase costs about one product.
//
// Babai (Eq. babai_update) is systolic over 8 warps: lane r holds row r of
// the CTA's 32, warp w holds coordinates [w CB, (w+1) CB) of the group
// (CB = g/8, resolved as sub-blocks of 8).  Warp 7 resolves its
// coordinates first and hands the code changes down through shared memory;
// warp w applies the column updates of every higher block in descending
// column order as they arrive, then resolves its own block from the top.
// Each u_l thus sees the same fused multiply-adds in the same order as the
// coordinate-by-coordinate recursion.  The change of the group objective
// (Eq. group_bils) is summed per warp and reduced over the warps per row; a
// proposal is kept iff it is finite and below zero (an unchanged row gives
// exactly zero).
//
// One CTA (832 threads):
//   warp 0        TMA producer (code tiles, digit tiles)
//   warp 1        TMEM allocation and the single-thread MMA issuer
//   warps 2..17   drain: digit sums -> double-float partial of T_i
//   warps 18..25  Babai: targets, proposals, acceptance, codes
// Cluster signals: two sets of counters in every CTA's shared memory, one
// counter per source CTA, which that CTA increments once per phase (remote
// reductions with release semantics at cluster scope; readers poll with
// acquire): `pcnt` -- the partials of the phase are in global memory;
// `ccnt` -- the codes of the phase are in Q and the code plane.  Phase i is
// complete when all four counters of a set reach i + 1.  (A single summed
// counter would not do: the CTAs may be a phase apart.)  Counters, unlike
// barrier phases, may be waited for out of order: the producer waits only
// in the phases where it holds the pending group.
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
constexpr int kStages = 2;
constexpr int kCluster = 4;            // CTAs per row tile
constexpr int kRows = 128 / kCluster;  // Babai rows per CTA (one per lane)
constexpr uint32_t kIdesc = tc::idesc_f16_f32(128, 256);
constexpr int kDrainWarps = 16;
constexpr int kBabaiWarps = 8;
constexpr int kDrain0 = 2;                         // first drain warp
constexpr int kBabai0 = kDrain0 + kDrainWarps;     // first Babai warp
constexpr int kThreads = 32 * (kBabai0 + kBabaiWarps);
constexpr int kBarDrain = 1, kBarBabai = 2;        // named barriers

// Packed rows of R_i (upper triangular, g x g): row l holds columns
// 16 floor(l/16) .. g-1, so every row starts on a 64-byte boundary.
__host__ __device__ constexpr int rpk_row_off(int l, int g) {
    return 16 * ((l >> 4) * g - 8 * (l >> 4) * ((l >> 4) - 1)) + (l & 15) * (g - 16 * (l >> 4));
}
__host__ __device__ constexpr int rpk_size(int g) { return rpk_row_off(g, g); }

// shared memory (g = 128 sizes; g = 64 uses less of each)
constexpr int kOffLo = kStages * kStage;                   // drain low parts [16][512]
constexpr int kOffRpk = kOffLo + 16 * 32 * kDrainWarps * 4;
constexpr int kOffYs = kOffRpk + rpk_size(128) * 4;        // targets / code changes [g][32]
constexpr int kOffCs = kOffYs + 128 * kRows * 4;           // codes [g/4][32] words
constexpr int kOffRow = kOffCs + 32 * kRows * 4;           // s, z, live of the 32 rows
constexpr int kOffFp = kOffRow + 3 * kRows * 4;            // dF parts [8 warps][32]
constexpr int kOffRd = kOffFp + kBabaiWarps * kRows * 4;   // 1 / R_ll [g]
constexpr int kOffUs = kOffRd + 128 * 4;                   // u stash [8 warps][8][32]
constexpr int kOffBar = kOffUs + kBabaiWarps * 8 * kRows * 4;
constexpr int kSmem = 1024 + kOffBar + 512;
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

// Shared-memory layout of the Babai exchange: per coordinate l a row of 32
// slots (one per Babai row r), the row index XOR-ed with l/4 so that both the
// target formation (a row per warp, l across lanes) and the systolic stage
// (l fixed, a row per lane) are free of bank conflicts.  Ys holds the
// targets y, then, once block w has consumed its own, that block's code
// changes.  Cs holds the current codes, four per word.
__device__ __forceinline__ int ys_idx(int l, int r) { return l * kRows + (r ^ ((l >> 2) & 31)); }
__device__ __forceinline__ int cs_idx(int k, int r) { return k * kRows + (r ^ (k & 31)); }

// Babai targets y = (Pt_i - sum of partials) / s of rows 4 bw .. 4 bw + 3 of
// the CTA's 32 (double-float until the subtraction is done), coalesced: a
// row at a time, NT consecutive coordinates per lane.  Also each row's codes
// and its scale, zero point and whether it takes a proposal.
template <int NT>
__device__ __forceinline__ void form_targets(const SweepArgs &a, float *Ys, uint32_t *Cs,
                                             float *rowS, int *rowZ, int *rowLive, int i,
                                             int bw, int lane, int jb, const float *th,
                                             const float *tl, bool ok) {
    constexpr int g = 32 * NT;
    constexpr int nks = kCluster / (g / 64);   // K parts of the phase product
    constexpr int per = kRows / kBabaiWarps;   // rows per Babai warp
    const int l0 = NT * lane;
#pragma unroll
    for (int rr = 0; rr < per; ++rr) {
        const int r = per * bw + rr;
        const int jr = jb + r;
        const int j = min(jr, a.p - 1);
        const float s = a.S[(size_t)j * a.G + i];
        const bool live = ok && jr < a.p && a.active[j] != 0 && fabsf(s) > a.eps;
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
#pragma unroll
        for (int sp = 0; sp < nks; ++sp) {
            const size_t o = ((size_t)sp * a.p_pad + j) * g + l0;
            float hv[NT], lv[NT];
            if constexpr (NT == 4) {
                const float4 h4 = __ldcg(reinterpret_cast<const float4 *>(th + o));
                const float4 l4 = __ldcg(reinterpret_cast<const float4 *>(tl + o));
                hv[0] = h4.x; hv[1] = h4.y; hv[2] = h4.z; hv[3] = h4.w;
                lv[0] = l4.x; lv[1] = l4.y; lv[2] = l4.z; lv[3] = l4.w;
            } else {
                const float2 h2 = __ldcg(reinterpret_cast<const float2 *>(th + o));
                const float2 l2 = __ldcg(reinterpret_cast<const float2 *>(tl + o));
                hv[0] = h2.x; hv[1] = h2.y;
                lv[0] = l2.x; lv[1] = l2.y;
            }
#pragma unroll
            for (int e = 0; e < NT; ++e) {
                const float sm = y[e] - hv[e];
                const float bb = sm - y[e];
                const float er = (y[e] - (sm - bb)) + (-hv[e] - bb);
                y[e] = sm;
                yl[e] += er - lv[e];
            }
        }
#pragma unroll
        for (int e = 0; e < NT; ++e) Ys[ys_idx(l0 + e, r)] = live ? (y[e] + yl[e]) / s : 0.f;
        if constexpr (NT == 4) {
            Cs[cs_idx(lane, r)] = *reinterpret_cast<const uint32_t *>(a.Q + off);
        } else {
            const uint32_t mine = *reinterpret_cast<const uint16_t *>(a.Q + off);
            const uint32_t next = __shfl_down_sync(0xffffffffu, mine, 1);
            if ((lane & 1) == 0) Cs[cs_idx(lane >> 1, r)] = mine | (next << 16);
        }
        if (lane == 0) {
            rowS[r] = s;
            rowZ[r] = a.Z[(size_t)j * a.G + i];
            rowLive[r] = live ? 1 : 0;
        }
    }
}

// Systolic Babai for group i of the CTA's 32 rows (row r = lane) on the CB
// coordinates of block w (Babai warp), from the targets and codes in Ys and
// Cs.  Rs: packed R_i; Rds: 1 / R_ll; Fp: per-warp dF parts [w][r]; blk: one
// flag per block, set to i + 1 when the block's code changes of phase i are
// in Ys.  ok: every earlier wait succeeded (else only the hand-off protocol
// is kept).
template <int NT>
__device__ __forceinline__ void babai_block(const SweepArgs &a, const float *Rs, float *Rds,
                                            float *Us, float *Ys, const uint32_t *Cs, const float *rowS,
                                            const int *rowZ, const int *rowLive, float *Fp,
                                            uint32_t *blk, int i, int w, int lane, int jb,
                                            bool ok) {
    constexpr int g = 32 * NT;
    constexpr int CB = g / kBabaiWarps;     // coordinates per warp (16 or 8)
    constexpr int NSB = CB / 8;             // sub-blocks of 8 coordinates
    const int c0 = w * CB;
    const int r = lane;
    const bool live = rowLive[r] != 0;
    // Rs[ro0 + tt rs + h] is R[c0 + tt][h]: the block's rows lie in one
    // 16-row band of the packed layout
    const int ro0 = rpk_row_off(c0, g) - 16 * (c0 >> 4);
    const int rs = g - 16 * (c0 >> 4);
    if (lane < CB) Rds[c0 + lane] = 1.0f / Rs[ro0 + lane * rs + c0 + lane];
    __syncwarp();
    float u[CB];
#pragma unroll
    for (int t = 0; t < CB; ++t) u[t] = Ys[ys_idx(c0 + t, r)];
    // column updates from every higher block, descending (per coordinate the
    // columns in descending order)
    for (int b = kBabaiWarps - 1; b > w; --b) {
        if (!tc::flag_wait(tc::smem_u32(blk + b), (uint32_t)(i + 1), b > w + 1)) ok = false;
        float dv[CB];
#pragma unroll
        for (int t = 0; t < CB; ++t) dv[t] = Ys[ys_idx(b * CB + t, r)];
#pragma unroll
        for (int tt = 0; tt < CB; ++tt) {
            float rv[CB];
#pragma unroll
            for (int k = 0; k < CB; k += 4) {
                const float4 v4 = *reinterpret_cast<const float4 *>(Rs + ro0 + tt * rs + b * CB + k);
                rv[k] = v4.x; rv[k + 1] = v4.y; rv[k + 2] = v4.z; rv[k + 3] = v4.w;
            }
#pragma unroll
            for (int t = CB - 1; t >= 0; --t) u[tt] = fmaf(-rv[t], dv[t], u[tt]);
        }
    }
    // own block, sub-blocks of 8 from the top (Eq. babai_update); the
    // change of the group objective is summed as coordinates become final
    // (Eq. group_bils).  While a sub-block resolves, the u of the lower ones
    // wait in shared memory (Us), which keeps the resolve in registers.
    uint32_t cw[CB / 4];   // current codes, four per word
#pragma unroll
    for (int k = 0; k < CB / 4; ++k) cw[k] = Cs[cs_idx(c0 / 4 + k, r)];
    auto qc = [&](int t) { return (float)((cw[t >> 2] >> (8 * (t & 3))) & 0xFFu); };
    const float qmaxf = (float)a.qmax;
    constexpr float kRound = 12582912.0f;   // 1.5 * 2^23: rounds to nearest even
    float *us = Us + w * (CB - 8) * kRows;   // [CB - 8][32] of this warp
#pragma unroll
    for (int t = 0; t < CB - 8; ++t) us[t * kRows + r] = u[t];
    float acc = 0.f;
#pragma unroll
    for (int sb = NSB - 1; sb >= 0; --sb) {
        const int s0 = 8 * sb;
        float v[8];   // u of this sub-block
#pragma unroll
        for (int t = 0; t < 8; ++t) v[t] = (sb == NSB - 1) ? u[s0 + t] : us[(s0 + t) * kRows + r];
        // tri[tt][t] = R[c0 + s0 + tt][c0 + s0 + t], t > tt
        float tri[8][8];
#pragma unroll
        for (int tt = 0; tt < 7; ++tt) {
#pragma unroll
            for (int k = tt & ~3; k < 8; k += 4) {
                const float4 v4 =
                    *reinterpret_cast<const float4 *>(Rs + ro0 + (s0 + tt) * rs + c0 + s0 + k);
                tri[tt][k] = v4.x; tri[tt][k + 1] = v4.y; tri[tt][k + 2] = v4.z; tri[tt][k + 3] = v4.w;
            }
        }
        // a row that takes no proposal: 1 / R_ll = 0 keeps x = q, no change
        float rd[8], dq[8];
#pragma unroll
        for (int t = 0; t < 8; ++t) rd[t] = live ? Rds[c0 + s0 + t] : 0.f;
#pragma unroll
        for (int t = 7; t >= 0; --t) {
            const float qf = qc(s0 + t);
            const float x = fmaf(v[t], rd[t], qf);
            const float qv = fminf(fmaxf(__fsub_rn(__fadd_rn(x, kRound), kRound), 0.f), qmaxf);
            dq[t] = qv - qf;
            // the next coordinate's update first: it is on the chain
            if (t > 0) v[t - 1] = fmaf(-tri[t - 1][t], dq[t], v[t - 1]);
#pragma unroll
            for (int tt = 0; tt + 1 < t; ++tt) v[tt] = fmaf(-tri[tt][t], dq[t], v[tt]);
        }
        // every u of the sub-block is final: its part of dF, then its changes
        // replace its targets
#pragma unroll
        for (int t = 7; t >= 0; --t) {
            const int l = c0 + s0 + t;
            const float yv = Ys[ys_idx(l, r)];
            const float av = Rs[ro0 + (s0 + t) * rs + l] * dq[t] - v[t];
            acc = fmaf(av - yv, av + yv, acc);
            Ys[ys_idx(l, r)] = dq[t];
        }
        // the lower sub-blocks of this block take this sub-block's columns
#pragma unroll
        for (int sl = 0; sl < sb; ++sl) {
#pragma unroll
            for (int tt = 0; tt < 8; ++tt) {
                float rv[8];
#pragma unroll
                for (int k = 0; k < 8; k += 4) {
                    const float4 v4 = *reinterpret_cast<const float4 *>(
                        Rs + ro0 + (8 * sl + tt) * rs + c0 + s0 + k);
                    rv[k] = v4.x; rv[k + 1] = v4.y; rv[k + 2] = v4.z; rv[k + 3] = v4.w;
                }
                float ul = us[(8 * sl + tt) * kRows + r];
#pragma unroll
                for (int t = 7; t >= 0; --t) ul = fmaf(-rv[t], dq[t], ul);
                us[(8 * sl + tt) * kRows + r] = ul;
            }
        }
    }
    __syncwarp();
    if (lane == 0) tc::flag_store_release(tc::smem_u32(blk + w), (uint32_t)(i + 1));
    Fp[w * kRows + r] = acc;
    // every block's dF part of this row
    tc::named_bar_sync(kBarBabai, 32 * kBabaiWarps);
    float F = 0.f;
#pragma unroll
    for (int b = kBabaiWarps - 1; b >= 0; --b) F += Fp[b * kRows + r];
    const float s = rowS[r];
    const float dF = s * s * F;
    const int jr = jb + r;
    if (ok && live && isfinite(dF) && dF < 0.f) {
        const int j = jr;
        const int z = rowZ[r];
        const size_t off = (size_t)j * a.d + i * g + c0;
        int qn[CB];
#pragma unroll
        for (int t = 0; t < CB; ++t) qn[t] = (int)qc(t) + (int)Ys[ys_idx(c0 + t, r)];
        uint32_t nw[CB / 4], hw[CB / 2];
#pragma unroll
        for (int k = 0; k < CB / 4; ++k)
            nw[k] = (uint32_t)qn[4 * k] | ((uint32_t)qn[4 * k + 1] << 8) |
                    ((uint32_t)qn[4 * k + 2] << 16) | ((uint32_t)qn[4 * k + 3] << 24);
#pragma unroll
        for (int k = 0; k < CB / 2; ++k)
            hw[k] = (uint32_t)__half_as_ushort(__int2half_rn(qn[2 * k] - z)) |
                    ((uint32_t)__half_as_ushort(__int2half_rn(qn[2 * k + 1] - z)) << 16);
        __half *crow = a.cplane + (size_t)j * a.d_pad + i * g + c0;
        if constexpr (CB == 16) {
            *reinterpret_cast<uint4 *>(a.Q + off) = make_uint4(nw[0], nw[1], nw[2], nw[3]);
            reinterpret_cast<uint4 *>(crow)[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            reinterpret_cast<uint4 *>(crow)[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
        } else {
            *reinterpret_cast<uint2 *>(a.Q + off) = make_uint2(nw[0], nw[1]);
            *reinterpret_cast<uint4 *>(crow) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        }
        if (w == 0) a.accepted[j] += 1;
    }
}

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
    float *Lo = (float *)(smem + kOffLo);
    float *Rs = (float *)(smem + kOffRpk);
    float *Ys = (float *)(smem + kOffYs);
    uint32_t *Cs = (uint32_t *)(smem + kOffCs);
    float *rowS = (float *)(smem + kOffRow);
    int *rowZ = (int *)(rowS + kRows);
    int *rowLive = rowZ + kRows;
    float *Fp = (float *)(smem + kOffFp);
    float *Rds = (float *)(smem + kOffRd);
    float *Us = (float *)(smem + kOffUs);
    uint64_t *bars = (uint64_t *)(smem + kOffBar);
    uint32_t *blk = (uint32_t *)(bars + 2 * kStages + 6);   // one flag per Babai block
    uint32_t *tmem_slot = blk + kBabaiWarps;
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    int *consumed = (int *)(tmem_slot + 2);
    uint32_t *counters = tmem_slot + 4;   // pcnt[4], ccnt[4]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int rank = (int)tc::cluster_ctarank();
    const int cpart = rank % ncol, kpart = rank / ncol;
    const int j0 = (blockIdx.x / kCluster) * 128;
    const int jb = j0 + kRows * rank;     // first of this CTA's Babai rows
    const int h0 = kpart * a.seg;
    const int nseg = max(0, min(a.G, h0 + a.seg) - h0);
    const int nchunks = nseg * nkc;

    auto full = [&](int s) { return tc::smem_u32(bars + s); };
    auto empty = [&](int s) { return tc::smem_u32(bars + kStages + s); };
    auto afull = [&](int b) { return tc::smem_u32(bars + 2 * kStages + b); };
    auto aempty = [&](int b) { return tc::smem_u32(bars + 2 * kStages + 2 + b); };
    const uint32_t lbar = tc::smem_u32(bars + 2 * kStages + 4);   // factor copy
    const uint32_t done = tc::smem_u32(bars + 2 * kStages + 5);
    const uint32_t pcnt = tc::smem_u32(counters);       // partials, one per source CTA
    const uint32_t ccnt = tc::smem_u32(counters + 4);   // codes, one per source CTA
    // phase i of every CTA of the cluster is out
    auto wait_all = [&](uint32_t base, int i) {
        bool ok = true;
#pragma unroll 1
        for (int k = 0; k < kCluster && ok; ++k) ok = tc::wait_count_cluster(base + 4 * k, i + 1);
        return ok;
    };
    // this CTA's phase is out, in every CTA of the cluster
    auto signal_all = [&](uint32_t base) {
        tc::fence_acq_rel_cluster();
        for (int r = 0; r < kCluster; ++r) tc::count_up_cluster(tc::map_cluster(base + 4 * rank, r));
    };
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
        for (int b = 0; b < kBabaiWarps; ++b) blk[b] = 0;
        for (int k = 0; k < 2 * kCluster; ++k) counters[k] = 0;
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
    // every CTA's counters are initialised before any CTA adds to them
    tc::cluster_sync();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // scales, active rows and codes come from the preceding kernels
    tc::pdl_wait();
    tc::pdl_launch_dependents();

    int cp = 0;               // producer: chunks issued
    int cm = 0;               // MMA issuer: chunks consumed
    int nl = 0;               // Babai leader: factor copies issued

    if (warp == 0 && lane == 0) {
        // ------------------------------------------------ producer
        for (int i = 0; i < a.G && !*abort_flag; ++i) {
            const int m0 = i * g + cpart * 64;    // first row of Ht (output column)
            const bool holds = i >= 1 && i - 1 >= h0 && i - 1 < h0 + nseg;
            // the folded projection of this CTA's Babai rows for group i,
            // read when the phase's targets are formed
            for (int r = 0; r < kRows && jb + r < a.p; ++r) {
                tc::prefetch_l2(a.pt_hi + (size_t)(jb + r) * a.d + i * g, g * sizeof(float));
                tc::prefetch_l2(a.pt_lo + (size_t)(jb + r) * a.d + i * g, g * sizeof(float));
            }
            for (int c = 0; c < nchunks; ++c) {
                const int u = c / nkc, kc = c % nkc;
                if (holds && u == nseg - 1 && kc == 0) {
                    // the last group is i-1: its codes from all four CTAs
                    if (!wait_all(ccnt, i - 1)) {
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
    } else if (warp >= kDrain0 && warp < kBabai0) {
        // ------------------------------------------------ drain
        const int q = warp & 3, cq = (warp - kDrain0) >> 2;   // lane quarter, 16-column quarter
        const int row = j0 + 32 * q + lane;
        const float *srow = a.S + (size_t)min(row, a.p - 1) * a.G;
        const int dw = warp - kDrain0;
        // low parts of this thread's 16 double-float accumulators
        float *lo = Lo + (threadIdx.x - 32 * kDrain0);
        int ud = 0;
        for (int i = 0; i < a.G; ++i) {
            float hi[16];
#pragma unroll
            for (int e = 0; e < 16; ++e) {
                hi[e] = 0.f;
                lo[e * 32 * kDrainWarps] = 0.f;
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
                        lo[(cc + e) * 32 * kDrainWarps] += e2 + fmaf(vl, scale, pe);
                    }
                }
                ++ud;
            }
            // partial of this CTA in slot i & 1; the slot's previous contents
            // (phase i-2) were read by every CTA's Babai warps before their
            // codes of phase i-2 went out
            if (ok && i >= 2 && !wait_all(ccnt, i - 2)) {
                ok = false;
                *abort_flag = 1;
            }
            float *th = a.t_hi + (size_t)(i & 1) * a.nks * a.p_pad * g;
            float *tl = a.t_lo + (size_t)(i & 1) * a.nks * a.p_pad * g;
            if (ok && row < a.p) {
                const size_t o = ((size_t)kpart * a.p_pad + row) * g + cpart * 64 + cq * 16;
#pragma unroll
                for (int e = 0; e < 16; e += 4) {
                    float x[4], y[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        two_sum(hi[e + k], lo[(e + k) * 32 * kDrainWarps], x[k], y[k]);
                    *reinterpret_cast<float4 *>(th + o + e) = make_float4(x[0], x[1], x[2], x[3]);
                    *reinterpret_cast<float4 *>(tl + o + e) = make_float4(y[0], y[1], y[2], y[3]);
                }
            }
            // each thread's partial is visible cluster-wide before the signal
            tc::fence_acq_rel_cluster();
            tc::named_bar_sync(kBarDrain, 32 * kDrainWarps);
            if (dw == 0 && lane == 0) signal_all(pcnt);
        }
    } else if (warp >= kBabai0) {
        // ------------------------------------------------ Babai
        const int bw = warp - kBabai0;
        if (bw == 0 && lane == 0) {
            // the factor of group 0
            tc::mbar_expect_tx(lbar, (uint32_t)(kRpk * sizeof(float)));
            tc::bulk_load(tc::smem_u32(Rs), a.Rpk, kRpk * sizeof(float), lbar);
            ++nl;
        }
        for (int i = 0; i < a.G; ++i) {
            // the partials of all four CTAs and the factor R_i
            bool ok = !*abort_flag;
            if (ok) ok = wait_all(pcnt, i);
            if (ok) ok = tc::mbar_wait(lbar, i & 1);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) *abort_flag = 1;
            const float *th = a.t_hi + (size_t)(i & 1) * a.nks * a.p_pad * g;
            const float *tl = a.t_lo + (size_t)(i & 1) * a.nks * a.p_pad * g;
            form_targets<NT>(a, Ys, Cs, rowS, rowZ, rowLive, i, bw, lane, jb, th, tl, ok);
            tc::named_bar_sync(kBarBabai, 32 * kBabaiWarps);
            babai_block<NT>(a, Rs, Rds, Us, Ys, Cs, rowS, rowZ, rowLive, Fp, blk, i, bw, lane, jb,
                            ok);
            // the accepted codes reach the other CTAs' tensor-map loads
            tc::fence_proxy_async_global();
            tc::fence_acq_rel_cluster();
            tc::named_bar_sync(kBarBabai, 32 * kBabaiWarps);
            if (bw == 0 && lane == 0) {
                signal_all(ccnt);
                // the next group's factor (every Babai warp is done with this one)
                if (i + 1 < a.G && !*abort_flag) {
                    tc::fence_proxy_async_smem();
                    tc::mbar_expect_tx(lbar, (uint32_t)(kRpk * sizeof(float)));
                    tc::bulk_load(tc::smem_u32(Rs), a.Rpk + (size_t)(i + 1) * kRpk,
                                  kRpk * sizeof(float), lbar);
                    ++nl;
                }
            }
        }
        if (bw == 0 && lane == 0 && nl > 0 && !tc::mbar_wait(lbar, (nl - 1) & 1)) *abort_flag = 1;
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
    tc::tc_fence_before();
    __syncwarp();
    // no CTA leaves while another may still add to its counters
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
