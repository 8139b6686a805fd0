// Gram matrices of the joint scale fit on the tensor cores, exact for the
// digit representation of H.
//
// Sec. 3.3.1, Eq. scale_design: Gram_j[i,h] = (A_i c_i)^T (A_h c_h)
// = c_i^T H_ih c_h with integer codes c = q - z.  Each g x g block H_ih is
// written as 2^(E_ih - 9) * sum_t a_t 2^(-10 t), t = 0..3, with integer
// digits |a_t| <= 512 (exact in fp16) and E_ih the block's exponent
// (max |H_ih| <= 2^E_ih), which represents every entry to within
// 2^(E_ih - 40).  The codes are fp16 as well (|c| <= 255), so
//     D_t[j, m] = sum_{k in grp h} c_j[k] a_t[k, m]
// is an integer below 128 * 255 * 512 < 2^24: every tensor-core partial sum
// is exact whatever the accumulator's rounding.  The epilogue forms the
// integer dots G_t = sum_{m in grp i} c_j[m] D_t[j, m] and
//     Gram_j[i,h] = 2^(E_ih - 9) (G_0 + G_1 2^-10 + G_2 2^-20 + G_3 2^-30)
// in float64.  Only h <= i is computed; the block is mirrored.  The pair of
// groups {i, G-1-i} of a 128-row tile holds G + 1 blocks; a CTA owns one of
// `nparts` contiguous ranges of them (the host picks nparts so that the
// CTAs fill the SMs' last wave).
//
// Roles: warp 0 TMA producer; warp 1 TMEM allocation and MMA issuer;
// warps 2..9 epilogue: warp w reads TMEM lanes 32 (w % 4) .. and 32 of the
// 64 columns of a unit; the two warps of a lane quarter add their partial
// dots through shared memory at the end of each block.  One unit of work is
// (h, column half of group i): 4 accumulators of 64 columns (one per digit
// plane), double-buffered in 512 TMEM columns.
#include <type_traits>

#include "df.cuh"
#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kTileA = 128 * 64 * 2;   // 128 code rows x 64 K (fp16)
constexpr int kTileB = 64 * 64 * 2;    // 64 H rows x 64 K, one digit plane (fp16)
constexpr int kStage = kTileA + 4 * kTileB;
// Codes of group i are staged per tile as int8 when they fit (|q - z| <= 127,
// up to 7 bits; then the freed shared memory holds a fourth pipeline stage)
// and as int16 otherwise.
template <bool WIDE>
struct GramCfg {
    using code_t = typename std::conditional<WIDE, int16_t, int8_t>::type;
    static constexpr int kStages = WIDE ? 3 : 4;
    static constexpr int kCodesBytes = 128 * 128 * (int)sizeof(code_t);
};
constexpr int kPartBytes = 2 * 4 * 128 * 8;  // int64 partial dots, double-buffered
template <bool WIDE>
constexpr int gram_smem() {
    return 1024 + GramCfg<WIDE>::kStages * kStage + GramCfg<WIDE>::kCodesBytes + kPartBytes + 256;
}
constexpr int kThreads = 320;
// one MMA covers the four digit planes: they are consecutive 64-row tiles
// in shared memory, and their accumulators consecutive 64-column blocks
constexpr uint32_t kIdesc = tc::idesc_f16_f32(128, 256);

struct GramArgs {
    const uint8_t *Q;
    const int32_t *Z;
    const int *expo;     // [G][G] block exponents E_ih
    const int *active;   // optional: rows whose Gram matrix is needed
    float2 *gram;        // [p][G][G] as float pairs (hi, lo) of the float64 value
    int *status;
    int p, d, g, G, d_pad;
    int nparts;          // block ranges per (row tile, group pair): blockIdx.z
};

__device__ __forceinline__ int exact_int(float x) {
    // x is an integer with |x| < 2^22: add 1.5 * 2^23 and read the low bits
    return __float_as_int(x + 12582912.0f) - 0x4B400000;
}

// WIDE: codes wider than 4 bits, |D_t| < 2^24 converted by cvt and 64-bit
// integer dots; otherwise |c| <= 15, |D_t| < 2^20 and every partial dot of
// 8 terms fits in 32 bits.
template <bool WIDE>
__global__ void __launch_bounds__(kThreads, 1)
    tc_gram_kernel(const __grid_constant__ CUtensorMap mapC, const __grid_constant__ CUtensorMap mapS,
                   GramArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    using code_t = typename GramCfg<WIDE>::code_t;
    constexpr int kStages = GramCfg<WIDE>::kStages;
    constexpr int kCodesBytes = GramCfg<WIDE>::kCodesBytes;
    code_t *codes = (code_t *)(smem + kStages * kStage);   // [128 rows][128]
    long long *part = (long long *)(smem + kStages * kStage + kCodesBytes);   // [2][4][128]
    uint64_t *bars = (uint64_t *)(smem + kStages * kStage + kCodesBytes + kPartBytes);
    uint32_t *tmem_slot = (uint32_t *)(bars + 2 * kStages + 4);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j0 = blockIdx.x * 128;
    const int G = a.G, g = a.g;
    const int nhalf = g / 64, nkc = g / 64;   // column halves of group i; K chunks per block

    {
        int mine = 0;
        if (threadIdx.x < 128 && j0 + (int)threadIdx.x < a.p)
            mine = a.active ? a.active[j0 + threadIdx.x] : 1;
        if (!__syncthreads_or(mine)) return;
    }
    // groups handled by this CTA and the unit list: for each group i (h = 0..i,
    // half = 0..nhalf-1), K chunks kc = 0..nkc-1 per unit
    const int i_lo = blockIdx.y, i_hi = G - 1 - blockIdx.y;
    const int ngrp = (i_lo == i_hi) ? 1 : 2;
    auto group_of = [&](int n) { return n == 0 ? i_lo : i_hi; };
    const int units0 = (i_lo + 1) * nhalf;
    const int nunits_pair = units0 + (ngrp == 2 ? (i_hi + 1) * nhalf : 0);
    // this CTA's blocks: [nblk z / nparts, nblk (z + 1) / nparts) of the pair's
    const int nblk = nunits_pair / nhalf;
    const int ub = (nblk * (int)blockIdx.z / a.nparts) * nhalf;
    const int nunits = (nblk * ((int)blockIdx.z + 1) / a.nparts) * nhalf - ub;
    auto unit = [&](int u, int &gi, int &h, int &half) {
        const int n = u < units0 ? 0 : 1;
        const int r = u < units0 ? u : u - units0;
        gi = group_of(n);
        h = r / nhalf;
        half = r % nhalf;
    };

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
            tc::mbar_init(aempty(b), 8);
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
        tc::prefetch_tmap(&mapS);
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int nchunks = nunits * nkc;

    if (warp == 0 && lane == 0) {
        // ---------------- producer: per chunk, codes of group h and 4 digit planes
        int issued = 0;
        for (int c = 0; c < nchunks; ++c) {
            const int s = c % kStages;
            if (!tc::mbar_wait(empty(s), ((c / kStages) & 1) ^ 1) || *abort_flag) {
                *abort_flag = 1;
                break;
            }
            int gi, h, half;
            unit(ub + c / nkc, gi, h, half);
            const int kx = h * g + (c % nkc) * 64;
            tc::mbar_expect_tx(full(s), kStage);
            tc::tma_load_2d(tileA(s), &mapC, full(s), kx, j0);
#pragma unroll
            for (int t = 0; t < 4; ++t)
                tc::tma_load_2d(tileB(s, t), &mapS, full(s), kx, t * a.d_pad + gi * g + half * 64);
            issued = c + 1;
        }
        for (int c = issued > kStages ? issued - kStages : 0; c < issued; ++c)
            if (!tc::mbar_wait(full(c % kStages), (c / kStages) & 1)) *abort_flag = 1;
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        for (int u = 0; u < nunits && !*abort_flag; ++u) {
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
        // ---------------- epilogue: exact integer dots with the codes of group i
        const int q = warp & 3, cw = (warp - 2) >> 2;   // lane quarter, 32-column slice
        const int rl = 32 * q + lane;           // row within the tile
        const int row = j0 + rl;
        int cur_g = -1, par = 0;
        bool dead = false;                      // a wait gave up: skip work, keep the pair barriers
        long long acc[4] = {0, 0, 0, 0};
        for (int u = 0; u < nunits; ++u) {
            int gi, h, half;
            unit(ub + u, gi, h, half);
            if (gi != cur_g) {
                // stage this warp's columns of group gi (row rl written by its own thread)
                __syncwarp();
                for (int hf = 0; hf < nhalf; ++hf) {
                    const int c0 = hf * 64 + cw * 32;
                    if (row < a.p) {
                        const int zz = a.Z[(size_t)row * G + gi];
                        const uint4 *src = reinterpret_cast<const uint4 *>(a.Q + (size_t)row * a.d + gi * g + c0);
                        for (int m16 = 0; m16 < 2; ++m16) {
                            const uint4 v = src[m16];
                            const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                            for (int k = 0; k < 16; ++k)
                                codes[rl * 128 + c0 + m16 * 16 + k] =
                                    (code_t)((int)((w4[k >> 2] >> (8 * (k & 3))) & 0xFFu) - zz);
                        }
                    } else {
                        for (int m = 0; m < 32; ++m) codes[rl * 128 + c0 + m] = 0;
                    }
                }
                __syncwarp();
                cur_g = gi;
            }
            const int b = u & 1;
            if (!dead) {
                bool w = tc::mbar_wait(afull(b), (u >> 1) & 1);
                w = __shfl_sync(0xffffffffu, w && !*abort_flag, 0);
                tc::tc_fence_after();
                if (!w) {
                    *abort_flag = 1;
                    dead = true;
                }
            }
            if (!dead) {
                const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + b * 256 + cw * 32;
                const code_t *crow = codes + rl * 128 + half * 64 + cw * 32;
                int cr[32];
                if constexpr (WIDE) {
#pragma unroll
                    for (int e = 0; e < 32; e += 8) {
                        const int4 pk = *reinterpret_cast<const int4 *>(crow + e);
                        const int w4[4] = {pk.x, pk.y, pk.z, pk.w};
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            cr[e + 2 * k] = (int)(int16_t)(w4[k] & 0xFFFF);
                            cr[e + 2 * k + 1] = w4[k] >> 16;
                        }
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 32; e += 16) {
                        const int4 pk = *reinterpret_cast<const int4 *>(crow + e);
                        const int w4[4] = {pk.x, pk.y, pk.z, pk.w};
#pragma unroll
                        for (int k = 0; k < 16; ++k)
                            cr[e + k] = (int)(int8_t)((w4[k >> 2] >> (8 * (k & 3))) & 0xFF);
                    }
                }
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    uint32_t v0[16], v1[16];
                    tc::tmem_ld16(base + t * 64, v0);
                    tc::tmem_ld16(base + t * 64 + 16, v1);
                    tc::tmem_wait_ld();
                    if (t == 3) {
                        // every digit of this unit is in registers
                        tc::tc_fence_before();
                        __syncwarp();
                        if (lane == 0) tc::mbar_arrive(aempty(b));
                    }
                    if (WIDE) {
                        long long p0 = 0, p1 = 0, p2 = 0, p3 = 0;
#pragma unroll
                        for (int e = 0; e < 16; e += 2) {
                            p0 += (long long)cr[e] * __float2int_rn(__uint_as_float(v0[e]));
                            p1 += (long long)cr[e + 1] * __float2int_rn(__uint_as_float(v0[e + 1]));
                            p2 += (long long)cr[16 + e] * __float2int_rn(__uint_as_float(v1[e]));
                            p3 += (long long)cr[17 + e] * __float2int_rn(__uint_as_float(v1[e + 1]));
                        }
                        acc[t] += (p0 + p1) + (p2 + p3);
                    } else {
                        int p0 = 0, p1 = 0, p2 = 0, p3 = 0;
#pragma unroll
                        for (int e = 0; e < 16; e += 2) {
                            p0 += cr[e] * exact_int(__uint_as_float(v0[e]));
                            p1 += cr[e + 1] * exact_int(__uint_as_float(v0[e + 1]));
                            p2 += cr[16 + e] * exact_int(__uint_as_float(v1[e]));
                            p3 += cr[17 + e] * exact_int(__uint_as_float(v1[e + 1]));
                        }
                        acc[t] += (long long)((p0 + p1) + (p2 + p3));
                    }
                }
            }
            if (half == nhalf - 1) {
                // the pair of warps of this lane quarter adds its partial dots
                long long *pp = part + (size_t)par * 4 * 128;
                if (cw == 1) {
#pragma unroll
                    for (int t = 0; t < 4; ++t) pp[t * 128 + rl] = acc[t];
                }
                asm volatile("bar.sync %0, 64;" ::"r"(1 + q) : "memory");
                if (cw == 0 && row < a.p && !dead) {
#pragma unroll
                    for (int t = 0; t < 4; ++t) acc[t] += pp[t * 128 + rl];
                    const int E = a.expo[gi * G + h];
                    double v;
                    if constexpr (!WIDE) {
                        // |acc_t| < 128 * 15 * 2^20 < 2^31: the digit sum is one
                        // exact 64-bit integer, converted with a single rounding
                        // (two float64 operations instead of eleven; float64 is a
                        // narrow pipe on this GPU)
                        const long long V = acc[0] * (1LL << 30) + acc[1] * (1LL << 20) +
                                            acc[2] * (1LL << 10) + acc[3];
                        v = __ll2double_rn(V) *
                            __longlong_as_double((long long)(E - 39 + 1023) << 52);
                    } else {
                        v = ldexp((double)acc[0] + ldexp((double)acc[1], -10) +
                                      ldexp((double)acc[2], -20) + ldexp((double)acc[3], -30),
                                  E - 9);
                    }
                    // stored once as the float pair the scale solve works on
                    const DF vp = split_double(v);
                    const float2 v2 = make_float2(vp.h, vp.l);
                    float2 *gr = a.gram + (size_t)row * G * G;
                    gr[(size_t)gi * G + h] = v2;
                    gr[(size_t)h * G + gi] = v2;
                }
#pragma unroll
                for (int t = 0; t < 4; ++t) acc[t] = 0;
                par ^= 1;
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

// Per g x g block of H: E = the exponent with max |H_blk| <= 2^E.  With
// `sym` the maximum also runs over the mirrored block (bh, bi), so that the
// exponent map is symmetric for a matrix that is not (the target projection
// reads the exponent of block (k, n) for the digits of entry (n, k)).
__global__ void block_exponent_kernel(const float *__restrict__ Hs, int *__restrict__ expo, int d,
                                      int g, int sym) {
    const int G = d / g, bi = blockIdx.y, bh = blockIdx.x;
    float mx = 0.f;
    for (int idx = threadIdx.x; idx < g * g; idx += blockDim.x) {
        const int r = idx / g, c = idx % g;
        mx = fmaxf(mx, fabsf(Hs[(size_t)(bi * g + r) * d + bh * g + c]));
        if (sym) mx = fmaxf(mx, fabsf(Hs[(size_t)(bh * g + r) * d + bi * g + c]));
    }
    for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    __shared__ float wm[32];
    if ((threadIdx.x & 31) == 0) wm[threadIdx.x >> 5] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
        float m = 0.f;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) m = fmaxf(m, wm[w]);
        int e = 0;
        if (m > 0.f) {
            frexpf(m, &e);     // m = f 2^e, f in [0.5, 1): |H| <= 2^e
        }
        expo[bi * G + bh] = e;
    }
}

// Digits of every entry of H for the two integer-digit schemes, from the
// block exponent E (max |H_blk| <= 2^E):
//  * dig8 (bf16, six planes, target projection): x = H 2^(7 - E) in
//    [-128, 128], a_0 = rint(x), a_t = rint(256 * remainder);
//  * dig10 (fp16, four planes, Gram): x = H 2^(9 - E) in [-512, 512],
//    a_0 = rint(x), a_t = rint(1024 * remainder).
__global__ void slice_kernel(const float *__restrict__ Hs, const int *__restrict__ expo,
                             __nv_bfloat16 *__restrict__ dig8, __half *__restrict__ dig10, int d,
                             int d_pad, int g) {
    const int G = d / g;
    const size_t n = (size_t)d * d;
    const size_t plane = (size_t)d_pad * d_pad;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int r = (int)(idx / d), c = (int)(idx % d);
        const int E = expo[(r / g) * G + c / g];
        const size_t off = (size_t)r * d_pad + c;
        float x = ldexpf(Hs[idx], 7 - E);
#pragma unroll
        for (int t = 0; t < 6; ++t) {
            const float dgt = rintf(x);
            dig8[t * plane + off] = __float2bfloat16_rn(dgt);
            x = (x - dgt) * 256.f;
        }
        if (!dig10) continue;
        x = ldexpf(Hs[idx], 9 - E);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            const float dgt = rintf(x);
            dig10[t * plane + off] = __float2half_rn(dgt);
            x = (x - dgt) * 1024.f;
        }
    }
}

// Digits of a double-float matrix M = hi + lo (not necessarily symmetric) in
// the Gram scheme: x = M 2^(9 - E) in [-512, 512] with E the block exponent,
// four fp16 planes base 2^10.  The low part enters before the remainder is
// scaled, so the digits represent hi + lo to 2^(E - 40).
__global__ void slice10_kernel(const float *__restrict__ hi, const float *__restrict__ lo,
                               const int *__restrict__ expo, __half *__restrict__ dig, int d,
                               int d_pad, int g) {
    const int G = d / g;
    const size_t n = (size_t)d * d;
    const size_t plane = (size_t)d_pad * d_pad;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (size_t)gridDim.x * blockDim.x) {
        const int r = (int)(idx / d), c = (int)(idx % d);
        const int E = expo[(r / g) * G + c / g];
        const size_t off = (size_t)r * d_pad + c;
        float x = ldexpf(hi[idx], 9 - E);
        const float xl = ldexpf(lo[idx], 9 - E);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            const float dgt = rintf(x);
            dig[t * plane + off] = __float2half_rn(dgt);
            x = x - dgt;
            if (t == 0) x += xl;
            x *= 1024.f;
        }
    }
}

}  // namespace

cudaError_t launch_slice10(const float *hi, const float *lo, int *expo, __half *dig, int d,
                           int d_pad, int g, cudaStream_t s) {
    const int G = d / g;
    block_exponent_kernel<<<dim3(G, G), 256, 0, s>>>(hi, expo, d, g, 0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    size_t n = (size_t)d * d;
    int blocks = (int)((n + 255) / 256);
    if (blocks > 16 * num_sms()) blocks = 16 * num_sms();
    slice10_kernel<<<blocks, 256, 0, s>>>(hi, lo, expo, dig, d, d_pad, g);
    return cudaGetLastError();
}

cudaError_t launch_slices(const float *Hs, int *expo, __nv_bfloat16 *dig8, __half *dig10, int d,
                          int d_pad, int g, cudaStream_t s) {
    const int G = d / g;
    block_exponent_kernel<<<dim3(G, G), 256, 0, s>>>(Hs, expo, d, g, 0);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    size_t n = (size_t)d * d;
    int blocks = (int)((n + 255) / 256);
    if (blocks > 16 * num_sms()) blocks = 16 * num_sms();
    slice_kernel<<<blocks, 256, 0, s>>>(Hs, expo, dig8, dig10, d, d_pad, g);
    return cudaGetLastError();
}

cudaError_t launch_slices8(const float *M, int *expo, __nv_bfloat16 *dig8, int d, int d_pad,
                           int g, cudaStream_t s) {
    const int G = d / g;
    block_exponent_kernel<<<dim3(G, G), 256, 0, s>>>(M, expo, d, g, 1);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    size_t n = (size_t)d * d;
    int blocks = (int)((n + 255) / 256);
    if (blocks > 16 * num_sms()) blocks = 16 * num_sms();
    slice_kernel<<<blocks, 256, 0, s>>>(M, expo, dig8, nullptr, d, d_pad, g);
    return cudaGetLastError();
}

cudaError_t launch_tc_gram(const CUtensorMap &mapC, const CUtensorMap &mapS, const uint8_t *Q,
                           const int32_t *Z, const int *expo, const int *active, float2 *gram,
                           int p, int p_pad, int d, int d_pad, int g, int bits, int *status,
                           cudaStream_t s) {
    static std::atomic<unsigned long long> attr_narrow{0}, attr_wide{0};
    cudaError_t e = set_max_dynamic_smem((const void *)tc_gram_kernel<false>, gram_smem<false>(),
                                         attr_narrow);
    if (e == cudaSuccess)
        e = set_max_dynamic_smem((const void *)tc_gram_kernel<true>, gram_smem<true>(), attr_wide);
    if (e != cudaSuccess) return e;
    const int G = d / g;
    // parts per (row tile, group pair), 1 to 4: the fewest waves of CTAs,
    // each wave as long as one part of the pair's blocks plus a fixed cost
    // of about 5 % of the whole pair
    const int nsm = num_sms();
    const long long ctas = (long long)(p_pad / 128) * ((G + 1) / 2);
    int nparts = 1;
    double best = 0.0;
    for (int n = 1; n <= 4 && n <= G + 1; ++n) {
        const long long waves = (ctas * n + nsm - 1) / nsm;
        const double t = (double)waves * (1.0 / n + 0.05);
        if (n == 1 || t < best - 1e-9) {
            best = t;
            nparts = n;
        }
    }
    GramArgs a{Q, Z, expo, active, gram, status, p, d, g, G, d_pad, nparts};
    dim3 grid(p_pad / 128, (G + 1) / 2, nparts);
    if (bits <= 4)
        tc_gram_kernel<false><<<grid, kThreads, gram_smem<false>(), s>>>(mapC, mapS, a);
    else
        tc_gram_kernel<true><<<grid, kThreads, gram_smem<true>(), s>>>(mapC, mapS, a);
    return cudaGetLastError();
}

}  // namespace jarq
