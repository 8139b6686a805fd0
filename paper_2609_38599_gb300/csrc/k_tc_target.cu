// Babai targets of one Gauss-Seidel phase on the tensor cores, exact to
// double-float accuracy (Sec. 3.3.2, Eqs. conditional_residual and
// babai_update).
//
// The target of group i is y = R_i^{-T} (H r)_i / s_i with r = w - D_s c.
// With the folded rows Ht_i = R_i^{-T} H[grp i, :] and Pt = R^{-T}-folded
// target projection (Pt_i = R_i^{-T} (H w)_i),
//     s_i y = Pt_i - sum_h s_h Ht_ih c_h,
// where c = q - z are the current codes (new for groups before i, previous
// for the rest).  This kernel forms T_i = sum_h s_h Ht_ih c_h; the Babai
// kernel subtracts it from Pt_i.  The codes are exact in fp16, and Ht is
// held in four fp16 digit planes base 2^10 per g x g block (block exponent
// E_ih, |digit| <= 512), so for each group h of K the four digit products
//     D_t[j, m] = sum_{k in grp h} c_j[k] a_t[m, k]
// are integers below 128 * 255 * 512 < 2^24, exact in the tensor-core
// accumulators.  Per group h the epilogue combines the digits in
// double-float, multiplies by s_jh 2^(E_ih - 9) and adds to a double-float
// accumulator, so T_i carries about 40 significant bits: the subtraction
// Pt_i - T_i, where the low-rank parts of H cancel, loses none of the
// precision float32 would.
//
// One CTA: 128 rows x 64 columns of group i over the groups of one K split.
//   warp 0       TMA producer: codes tile + its share of the digit tiles
//   warp 1       TMEM allocation and the single-thread MMA issuer
//   warps 2..17  drain: warp w reads TMEM lanes 32 (w % 4) and 16 columns
// Four 64-column accumulators per group h, double-buffered (512 columns).
// The drain does 17 float32 operations per output and group, hence
// sixteen drain warps; the scale and block exponent of the next group are
// loaded one group ahead.
#include <cmath>

#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kTileA = 128 * 64 * 2;   // codes: 128 rows x 64 K, fp16
constexpr int kTileB = 64 * 64 * 2;    // one digit plane: 64 rows of Ht x 64 K
constexpr int kStage = kTileA + 4 * kTileB;
constexpr int kStages = 4;
constexpr int kSmem = 1024 + kStages * kStage + 256;
// one MMA covers the four digit planes: they are consecutive 64-row tiles
// in shared memory, and their accumulators consecutive 64-column blocks
constexpr uint32_t kIdesc = tc::idesc_f16_f32(128, 256);
constexpr int kDrainWarps = 16;
constexpr int kThreads = 32 * (2 + kDrainWarps);

struct TargetArgs {
    float *out_hi, *out_lo;   // [nsplit][p_pad][g]
    const float *S;           // [p][G]
    const int *expoT;         // [G][G] block exponents of Ht
    const int *active;        // optional: rows still refined
    int *status;
    int p, p_pad, d_pad, g, G, i, seg_per_split;
    int row0;                 // first row of this launch's tiles (a multiple of 128)
    float round_c;            // 1.5 * 2^(23 - k): rounds to multiples of 2^-k
};

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e) {
    s = a + b;
    const float bb = s - a;
    e = (a - (s - bb)) + (b - bb);
}

__global__ void __launch_bounds__(kThreads, 1)
    tc_target_kernel(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapT,
                     TargetArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *bars = (uint64_t *)(smem + kStages * kStage);
    uint32_t *tmem_slot = (uint32_t *)(bars + 2 * kStages + 4);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j0 = a.row0 + blockIdx.x * 128;
    const int m0 = a.i * a.g + blockIdx.y * 64;          // first row of Ht (output column)
    const int h0 = blockIdx.z * a.seg_per_split;
    const int h1 = min(a.G, h0 + a.seg_per_split);
    const int nkc = a.g / 64;

    auto full = [&](int s) { return tc::smem_u32(bars + s); };
    auto empty = [&](int s) { return tc::smem_u32(bars + kStages + s); };
    auto afull = [&](int b) { return tc::smem_u32(bars + 2 * kStages + b); };
    auto aempty = [&](int b) { return tc::smem_u32(bars + 2 * kStages + 2 + b); };
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
        *abort_flag = 0;
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
    // The previous grid (the Babai step of group i - 1) rewrites only the
    // codes of group i - 1, and reads the phase partials this grid writes.
    // Without the early stop (no active flags to read) each role therefore
    // waits for it only where it must: the producer before the code tile of
    // a chunk of group i - 1, the drain before writing the partials.  The
    // Ht digit tiles, the other code tiles and the scales do not change
    // during the sweep, so the products of the other groups can run while
    // the previous grid finishes.  With the early stop every thread waits
    // here, before reading the flags; so it does in the first phase, whose
    // previous grid is the scale solve that writes the scales.
    const bool early = !a.active && a.i > 0;
    if (!early) tc::pdl_wait();
    // The next grid (Babai of group i) is released at once: before its own
    // wait it reads nothing that this grid or the previous one writes.
    tc::pdl_launch_dependents();
    // a tile none of whose rows is still active (early stop, App. E) does
    // no work: the Babai step reads the partials of active rows only
    const bool live = early ? j0 < a.p
                            : __syncthreads_or(threadIdx.x < 128 && j0 + (int)threadIdx.x < a.p &&
                                               (!a.active || a.active[j0 + threadIdx.x] != 0));
    const int nseg = live ? max(0, h1 - h0) : 0;
    const int nchunks = nseg * nkc;

    if (warp == 0 && lane == 0) {
        // ---------------- producer
        int issued = 0;
        bool waited = !early;
        for (int c = 0; c < nchunks; ++c) {
            const int s = c % kStages;
            if (!tc::mbar_wait(empty(s), ((c / kStages) & 1) ^ 1) || *abort_flag) {
                *abort_flag = 1;
                break;
            }
            const int kx = h0 * a.g + c * 64;
            if (!waited && h0 + c / nkc == a.i - 1) {
                tc::pdl_wait();   // the codes of group i - 1
                waited = true;
            }
            tc::mbar_expect_tx(full(s), kStage);
            tc::tma_load_2d(tileA(s), &mapC, full(s), kx, j0);
#pragma unroll
            for (int t = 0; t < 4; ++t)
                tc::tma_load_2d(tileB(s, t), &mapT, full(s), kx, t * a.d_pad + m0);
            issued = c + 1;
        }
        // do not leave before the MMAs have consumed the stages filled here:
        // no copy or commit is in flight afterwards
        for (int c = issued > kStages ? issued - kStages : 0; c < issued; ++c)
            if (!tc::mbar_wait(empty(c % kStages), (c / kStages) & 1)) *abort_flag = 1;
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer: one unit per group h
        for (int u = 0; u < nseg && !*abort_flag; ++u) {
            const int b = u & 1;
            if (!tc::mbar_wait(aempty(b), ((u >> 1) & 1) ^ 1)) {
                *abort_flag = 1;
                break;
            }
            tc::tc_fence_after();
            for (int kc = 0; kc < nkc; ++kc) {
                const int c = u * nkc + kc;
                const int s = c % kStages;
                if (!tc::mbar_wait(full(s), (c / kStages) & 1) || *abort_flag) {
                    *abort_flag = 1;
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
            }
            tc::mma_commit(afull(b));
        }
    } else if (warp >= 2) {
        // ---------------- drain: digits -> double-float x s_h 2^(E - 9) -> accumulator
        const int q = warp & 3, cq = (warp - 2) >> 2;    // lane quarter, 16-column quarter
        const int row = j0 + 32 * q + lane;
        float hi[16], lo[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
            hi[e] = 0.f;
            lo[e] = 0.f;
        }
        bool ok = true;
        const float *srow = a.S + (size_t)min(row, a.p - 1) * a.G;
        const int *erow = a.expoT + (size_t)a.i * a.G;
        float s_next = nseg > 0 ? srow[h0] : 0.f;
        int e_next = nseg > 0 ? erow[h0] : 0;
        for (int u = 0; u < nseg; ++u) {
            const int b = u & 1, h = h0 + u;
            const float s_cur = row < a.p ? s_next : 0.f;
            const int e_cur = e_next;
            if (u + 1 < nseg) {
                s_next = srow[h + 1];
                e_next = erow[h + 1];
            }
            bool w = tc::mbar_wait(afull(b), (u >> 1) & 1);
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
                    // D_0 + D_1 2^-10 exactly as (vh, vl): the digit sums are
                    // integers with |D_0| <= 128 qmax 512 and |D_1 2^-10| < 2^14;
                    // t = D_1 2^-10 rounded to a multiple of 2^-k (by adding
                    // and subtracting 1.5 2^(23-k)), with k chosen on the host
                    // so that |D_0 + t| < 2^(24-k): then vh = D_0 + t and
                    // vl = D_1 2^-10 - t (|vl| <= 2^-(k+1)) are exact.  The
                    // D_2, D_3 terms are below 2^-20 of the sum and enter the
                    // low part.
                    float s2, e2;
                    const float d1 = __uint_as_float(v1[e]);
                    const float tq = __fsub_rn(__fmaf_rn(d1, 0x1p-10f, a.round_c), a.round_c);
                    const float vh = __fadd_rn(__uint_as_float(v0[e]), tq);
                    float vl = __fmaf_rn(d1, 0x1p-10f, -tq);
                    vl = fmaf(__uint_as_float(v2[e]), 0x1p-20f, vl);
                    vl = fmaf(__uint_as_float(v3[e]), 0x1p-30f, vl);
                    // (vh + vl) * scale, added to the accumulator
                    const float ph = vh * scale;
                    const float pe = fmaf(vh, scale, -ph);
                    two_sum(hi[cc + e], ph, s2, e2);
                    hi[cc + e] = s2;
                    lo[cc + e] += e2 + fmaf(vl, scale, pe);
                }
            }
        }
        // the previous grid reads the partials this drain overwrites
        if (early) tc::pdl_wait();
        if (ok && row < a.p) {
            const size_t o = (size_t)blockIdx.z * a.p_pad * a.g + (size_t)row * a.g + blockIdx.y * 64 + cq * 16;
#pragma unroll
            for (int e = 0; e < 16; e += 4) {
                float x[4], y[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) two_sum(hi[e + k], lo[e + k], x[k], y[k]);
                *reinterpret_cast<float4 *>(a.out_hi + o + e) = make_float4(x[0], x[1], x[2], x[3]);
                *reinterpret_cast<float4 *>(a.out_lo + o + e) = make_float4(y[0], y[1], y[2], y[3]);
            }
        }
    }
    tc::tc_fence_before();
    __syncwarp();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, ST_TIMEOUT);
}

}  // namespace

// Split of the K range (groups) over CTAs so that the launch covers the SMs.
int target_splits(int p_pad, int g, int G) {
    const int tiles = (p_pad / 128) * (g / 64);
    int n = num_sms() / tiles;
    if (n < 1) n = 1;
    if (n > kMaxSplit) n = kMaxSplit;
    if (n > G) n = G;
    return n;
}

cudaError_t launch_tc_target(const CUtensorMap &mapC, const CUtensorMap &mapT, float *out_hi,
                             float *out_lo, const float *S, const int *expoT, const int *active,
                             int p, int p_pad, int d_pad, int g, int G, int i, int nsplit,
                             int row0, int nrows, int qmax, int *status, cudaStream_t s,
                             bool pdl) {
    static std::atomic<unsigned long long> attr_done{0};
    const cudaError_t e = set_max_dynamic_smem((const void *)tc_target_kernel, kSmem, attr_done);
    if (e != cudaSuccess) return e;
    const int per = (G + nsplit - 1) / nsplit;
    if (row0 % 128 != 0 || nrows < 0 || row0 + nrows > p_pad) return cudaErrorInvalidValue;
    const int tiles = (nrows + 127) / 128;
    if (tiles == 0) return cudaSuccess;
    // quantum 2^-k of the exact digit split: the largest k with
    // 128 qmax 512 + 2^14 <= 2^(24-k)
    if (qmax < 1 || qmax > 255 || g > 128) return cudaErrorInvalidValue;
    const double bound = 128.0 * qmax * 512.0 + 16384.0;
    int kq = 0;
    while (kq < 7 && bound <= std::ldexp(1.0, 24 - (kq + 1))) ++kq;
    const float round_c = (float)std::ldexp(1.5, 23 - kq);
    TargetArgs a{out_hi, out_lo, S, expoT, active, status, p, p_pad, d_pad, g, G, i, per,
                 row0, round_c};
    dim3 grid(tiles, g / 64, nsplit);
    return launch_k(tc_target_kernel, grid, dim3(kThreads), (size_t)kSmem, s, pdl, mapC, mapT, a);
}

}  // namespace jarq
