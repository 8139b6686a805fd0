// Calibration Hessian accumulation H += scale * X^T X from fp16 activations
// on the tensor cores.  The H-form uses H = A^T A for the augmented design
// A = [X~; nu I] of Eq. strict_target, i.e. H = X~^T X~ + nu^2 I (App.
// "Propagation-Corrected Targets and QEP" writes it out); this entry point
// forms the X~^T X~ part (nu^2 I is added when the Hessian is prepared).  The
// paper forms its products from FP16 activations in FP32 (App. "Metrics");
// here every fp16 x fp16 product is exact and the sums are float32.
//
// X is read as it is produced, token-major [n][d], with no transpose: a TMA
// box of 64 tokens x 64 features lands as 64 rows of 128 bytes (128-byte
// swizzle), which is the MN-major operand layout of tcgen05.mma (MN =
// features, contiguous; K = tokens, 128 bytes apart; 8-token atoms 1024
// bytes apart; 64-feature atoms one box, 8 KiB, apart).
//
// One CTA computes one 128 x 256 tile (rows r0.., columns c0..) of the upper
// triangle of X^T X over all n tokens:
//   warp 0      TMA producer, 4-stage ring of 64-token chunks
//               (A: 128 features, B: 256 features; a diagonal tile whose A
//               features lie inside B reads them from B's tile)
//   warp 1      TMEM allocation and the single-thread MMA issuer: one
//               M128 x N256 x K16 MMA per 16 tokens
//   warps 2..9  drain: every 512 tokens the TMEM accumulator (restarted at
//               zero, two of them alternate) is added into float32
//               registers.  At the end the tile is added to H twice with
//               coalesced accesses: mirrored, H[col][row], straight from the
//               registers (a warp's 32 rows are contiguous there), and as
//               H[row][col] in float4 through shared memory.
// Each unordered pair {i, j} belongs to exactly one tile element with
// col >= row, so every element of H is written exactly once.
#include <math.h>

#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kBox = 64 * 64 * 2;          // one TMA box: 64 tokens x 64 features, fp16
constexpr int kTileA = 2 * kBox;           // 128 features
constexpr int kTileB = 4 * kBox;           // 256 features
constexpr int kStage = kTileA + kTileB;
constexpr int kStages = 4;
constexpr int kBars = 2 * kStages + 5;     // full, empty, afull[2], aempty[2], done
constexpr int kSmem = 1024 + kStages * kStage + 8 * kBars + 16;
constexpr int kChunksPerDrain = 8;         // 512 tokens per tensor-core sum
constexpr int kThreads = 320;
constexpr int kTld = 257;                  // row pitch (floats) of the staged tile
static_assert(128 * kTld * 4 <= kStages * kStage, "staged tile must fit the stage ring");

// fp16 x fp16 -> f32, M = 128, N = 256, both operands MN-major.
constexpr uint32_t kIdesc = tc::idesc_f16_f32(128, 256) | (1u << 15) | (1u << 16);

__device__ int g_syrk_status;

// Descriptor of an MN-major operand written by TMA with 128-byte swizzle:
// 64 contiguous MN elements per 128-byte row, K rows 128 bytes apart,
// 8-row atoms SBO = 1024 bytes apart along K, 64-element MN atoms
// LBO = 8192 bytes (one box) apart along MN.
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)(kBox >> 4) << 16;           // leading byte offset: next 64 features
    d |= (uint64_t)(1024 >> 4) << 32;           // stride byte offset: next 8 tokens
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

struct SyrkArgs {
    float *H;
    float scale;
    int d, n;
    int ct;          // column tiles of 256
    int rt;          // row tiles of 128
};

// Linear index of an upper tile -> (row tile, column tile); column tile cj
// holds row tiles 0 .. min(rt, 2 cj + 2) - 1.
__device__ __forceinline__ void tile_of(int t, int rt, int ct, int &ri, int &cj) {
    cj = 0;
    for (; cj < ct; ++cj) {
        const int m = min(rt, 2 * cj + 2);
        if (t < m) break;
        t -= m;
    }
    ri = t;
}

// One pass of the tile update H += scale * T over 256 threads, as float4
// read-modify-writes of H with 8 loads in flight per thread.  MIRROR false:
// H[r0+i][c0+j] for c0+j >= r0+i (float4 along j, 128 rows x 64); MIRROR
// true: H[c0+j][r0+i] for c0+j > r0+i (float4 along i, 256 rows x 32).  A
// float4 that straddles the diagonal updates its own elements only.
template <bool MIRROR>
__device__ __forceinline__ void add_tile_pass(const SyrkArgs &a, const float *T, int t, int r0,
                                              int c0) {
    constexpr int kSh = MIRROR ? 5 : 6;           // float4 per H row segment: 32 or 64
#pragma unroll 1
    for (int k0 = 0; k0 < 32; k0 += 8) {
        float4 h[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int idx = t + 256 * (k0 + k);
            const int u = idx >> kSh, v4 = 4 * (idx & ((1 << kSh) - 1));
            const int hr = MIRROR ? c0 + u : r0 + u, hc = MIRROR ? r0 + v4 : c0 + v4;
            // all four elements on the kept side of the diagonal
            const bool full = hr < a.d && hc < a.d && (MIRROR ? hr > hc + 3 : hc >= hr);
            h[k] = full ? *reinterpret_cast<const float4 *>(a.H + (size_t)hr * a.d + hc)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int idx = t + 256 * (k0 + k);
            const int u = idx >> kSh, v4 = 4 * (idx & ((1 << kSh) - 1));
            const int hr = MIRROR ? c0 + u : r0 + u, hc = MIRROR ? r0 + v4 : c0 + v4;
            if (hr >= a.d || hc >= a.d) continue;
            // tile element of H[hr][hc + m]
            auto tv = [&](int m) {
                return MIRROR ? T[(v4 + m) * kTld + u] : T[u * kTld + v4 + m];
            };
            float *hp = a.H + (size_t)hr * a.d + hc;
            if (MIRROR ? hr > hc + 3 : hc >= hr) {
                float4 v = h[k];
                v.x = fmaf(a.scale, tv(0), v.x);
                v.y = fmaf(a.scale, tv(1), v.y);
                v.z = fmaf(a.scale, tv(2), v.z);
                v.w = fmaf(a.scale, tv(3), v.w);
                *reinterpret_cast<float4 *>(hp) = v;
            } else {
                for (int m = 0; m < 4; ++m)
                    if (MIRROR ? hr > hc + m : hc + m >= hr) hp[m] = fmaf(a.scale, tv(m), hp[m]);
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads, 1)
    tc_syrk_kernel(const __grid_constant__ CUtensorMap mapX, SyrkArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *bars = (uint64_t *)(smem + kStages * kStage);
    uint32_t *tmem_slot = (uint32_t *)(bars + kBars);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int ri, cj;
    tile_of(blockIdx.x, a.rt, a.ct, ri, cj);
    const int r0 = ri * 128, c0 = cj * 256;
    const bool a_in_b = r0 >= c0 && r0 < c0 + 256;
    const int nchunks = (a.n + 63) / 64;
    const int nper = (nchunks + kChunksPerDrain - 1) / kChunksPerDrain;

    auto full = [&](int s) { return tc::smem_u32(bars + s); };
    auto empty = [&](int s) { return tc::smem_u32(bars + kStages + s); };
    auto afull = [&](int b) { return tc::smem_u32(bars + 2 * kStages + b); };
    auto aempty = [&](int b) { return tc::smem_u32(bars + 2 * kStages + 2 + b); };
    const uint32_t done = tc::smem_u32(bars + 2 * kStages + 4);
    auto tileB = [&](int s) { return tc::smem_u32(smem + s * kStage + kTileA); };
    auto tileA = [&](int s) {
        return a_in_b ? tileB(s) + (uint32_t)((r0 - c0) / 64) * kBox : tc::smem_u32(smem + s * kStage);
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(full(s), 1);
            tc::mbar_init(empty(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::mbar_init(afull(b), 1);
            tc::mbar_init(aempty(b), 8);
        }
        tc::mbar_init(done, 1);
        *abort_flag = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(tc::smem_u32(tmem_slot), 512);
        tc::tmem_relinquish();
    }
    if (warp == 0 && lane == 0) tc::prefetch_tmap(&mapX);
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- producer
            int issued = 0;
            for (int c = 0; c < nchunks; ++c) {
                const int s = c % kStages;
                if (!tc::mbar_wait(empty(s), ((c / kStages) & 1) ^ 1) || *abort_flag) {
                    *abort_flag = 1;
                    break;
                }
                tc::mbar_expect_tx(full(s), a_in_b ? kTileB : kStage);
                if (!a_in_b)
                    for (int m = 0; m < 2; ++m)
                        tc::tma_load_2d(tc::smem_u32(smem + s * kStage) + m * kBox, &mapX,
                                        full(s), r0 + 64 * m, c * 64);
                for (int m = 0; m < 4; ++m)
                    tc::tma_load_2d(tileB(s) + m * kBox, &mapX, full(s), c0 + 64 * m, c * 64);
                issued = c + 1;
            }
            // leave no copy in flight
            for (int c = issued > kStages ? issued - kStages : 0; c < issued; ++c)
                if (!tc::mbar_wait(full(c % kStages), (c / kStages) & 1)) *abort_flag = 1;
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer: accumulator b = per & 1 for each 512 tokens
            for (int per = 0; per < nper && !*abort_flag; ++per) {
                const int b = per & 1;
                if (!tc::mbar_wait(aempty(b), ((per >> 1) & 1) ^ 1)) {
                    *abort_flag = 1;
                    break;
                }
                tc::tc_fence_after();
                const int cbeg = per * kChunksPerDrain;
                const int cend = min(nchunks, cbeg + kChunksPerDrain);
                bool ok = true;
                for (int c = cbeg; c < cend; ++c) {
                    const int s = c % kStages;
                    if (!tc::mbar_wait(full(s), (c / kStages) & 1) || *abort_flag) {
                        ok = false;
                        break;
                    }
                    tc::tc_fence_after();
#pragma unroll
                    for (int sub = 0; sub < 4; ++sub) {
                        // 16 tokens = two 8-token atoms = 2048 bytes along K
                        const uint64_t ad = sdesc_mn_sw128(tileA(s)) + (uint64_t)(128 * sub);
                        const uint64_t bd = sdesc_mn_sw128(tileB(s)) + (uint64_t)(128 * sub);
                        tc::mma_bf16(tmem + b * 256, ad, bd, kIdesc, (c > cbeg || sub > 0) ? 1u : 0u);
                    }
                    tc::mma_commit(empty(s));
                }
                if (!ok) {
                    *abort_flag = 1;
                    break;
                }
                tc::mma_commit(afull(b));
            }
            // every MMA issued has finished before TMEM is released
            tc::mma_commit(done);
            if (!tc::mbar_wait(done, 0)) *abort_flag = 1;
        }
    } else {
        // ---------------- drain: TMEM -> float32 registers
        const int q = warp & 3, half = (warp - 2) >> 2;
        float acc[128];
#pragma unroll
        for (int e = 0; e < 128; ++e) acc[e] = 0.f;
        for (int per = 0; per < nper; ++per) {
            const int b = per & 1;
            bool w = tc::mbar_wait(afull(b), (per >> 1) & 1);
            w = __shfl_sync(0xffffffffu, w, 0) && !*abort_flag;
            if (!__all_sync(0xffffffffu, w)) {
                if (lane == 0) *abort_flag = 1;
                break;
            }
            tc::tc_fence_after();
            const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + b * 256 + half * 128;
#pragma unroll
            for (int cc = 0; cc < 128; cc += 32) {
                uint32_t v[32];
                tc::tmem_ld32(base + cc, v);
                tc::tmem_wait_ld();
#pragma unroll
                for (int e = 0; e < 32; ++e) acc[cc + e] += __uint_as_float(v[e]);
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(aempty(b));
        }
        // the stage ring is idle once the last accumulator has been read:
        // stage the tile as T[row][col]
        float *T = (float *)smem;
        if (!*abort_flag) {
            const int i = 32 * q + lane;
#pragma unroll
            for (int e = 0; e < 128; ++e) T[i * kTld + half * 128 + e] = acc[e];
        }
        asm volatile("bar.sync 1, 256;" ::: "memory");
        if (!*abort_flag) {
            const int t = threadIdx.x - 64;
            // H[row][col] for col >= row: a tile row is 64 float4 of H's row
            add_tile_pass<false>(a, T, t, r0, c0);
            // H[col][row] for col > row: a tile column is 32 float4 of H's row `col`
            add_tile_pass<true>(a, T, t, r0, c0);
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, 512);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicOr(&g_syrk_status, ST_TIMEOUT);
}

// Number of 128 x 256 tiles that meet the upper triangle of a d x d matrix.
int syrk_tiles(int d) {
    const int rt = (d + 127) / 128, ct = (d + 255) / 256;
    int n = 0;
    for (int cj = 0; cj < ct; ++cj) n += min(rt, 2 * cj + 2);
    return n;
}

}  // namespace
}  // namespace jarq

using namespace jarq;

extern "C" jarq_status jarq_accumulate_hessian(const void *X, int n, int d, float scale, float *H,
                                               void *stream) {
    if (n < 0 || d < 8 || d % 8 || d > 65536 || !isfinite(scale)) return JARQ_ERR_ARG;
    if (!H || !on_device(H) || ((uintptr_t)H & 15)) return JARQ_ERR_ARG;
    if (n == 0) return JARQ_OK;
    if (!X || !on_device(X) || ((uintptr_t)X & 15)) return JARQ_ERR_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    CUtensorMap map;
    if (make_tmap_f16(&map, X, (uint64_t)n, (uint64_t)d, 64) != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_ARG;
    }
    int *status = nullptr;
    int host = 0;
    cudaError_t e = cudaGetSymbolAddress((void **)&status, g_syrk_status);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(tc_syrk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem);
    if (e == cudaSuccess) e = cudaMemsetAsync(status, 0, sizeof(int), st);
    if (e == cudaSuccess) {
        SyrkArgs args{H, scale, d, n, (d + 255) / 256, (d + 127) / 128};
        ProfScope ps("syrk", st);
        tc_syrk_kernel<<<syrk_tiles(d), kThreads, kSmem, st>>>(map, args);
        e = cudaGetLastError();
        ps.done();
        count_launches(1);
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(&host, status, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    prof_collect();
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_CUDA;
    }
    return host ? JARQ_ERR_TIMEOUT : JARQ_OK;
}
