// Residual products (H r) on the tensor cores (tcgen05 + TMA), split precision.
//
// The residual r = w - D_s (q - z) (Eq. quantized_group) and the symmetric
// Hessian H are both split exactly into three bf16 planes,
// x = x1 + x2 + x3 (truncation splits of the float32 value), and
//     H r ~= sum over the six products r_a H_b with a + b <= 4
// (a, b = 1..3; the three dropped products are below float32 resolution),
// accumulated in float32.  Tensor-core accumulation truncates, so its error
// grows with the number of products summed into one accumulator; the kernel
// therefore (a) keeps the leading product r_1 H_1 and the five small products
// in separate TMEM accumulators, and (b) drains both into float32 registers
// (round to nearest) every 128 columns of K, restarting the TMEM sums at zero.
// Two accumulator pairs alternate so the MMAs of one 128-wide K period overlap
// the drain of the previous one.  Used for
//   * the full product H r at the start of an iteration (objective of
//     Eq. bbmils_columns and the scale gradient c_i^T (H r)_i), and
//   * the per-group phase product (H r)_i of the Gauss-Seidel sweep
//     (Eq. conditional_residual), split over K across CTAs.
//
// One CTA computes a 128-row x BN-column output tile:
//   warp 0      TMA producer: 3 A planes + 3 B planes per 64-wide K chunk
//   warp 1      TMEM allocation and the single-thread MMA issuer
//   warps 2..9  drain (TMEM -> register sums) and store (float32); warp w
//               reads TMEM lanes 32 (w % 4) .. + 31 and half (w - 2) / 4 of
//               the tile's columns
// Operands are K-major: A = r planes [3][p_pad][d_pad], B = H planes
// [3][d_pad][d_pad] (H symmetric, so row n of H is column n), both loaded
// with 128-byte swizzle.
#include "tc_common.cuh"

namespace jarq {
namespace {

constexpr int kTileA = 128 * 64 * 2;  // bytes of one 128 x 64 bf16 A tile
constexpr int kProducts = 8;
constexpr int kPeriod = 1;            // 64-wide K chunks per drain period
constexpr int kGroupRows = 8;         // row tiles per band in the full-product tile order
// (A plane, B plane) of each product, smallest first; the last, (0, 0), is
// the leading one.
__host__ __device__ constexpr int prod_a(int k) {
    constexpr int t[8] = {2, 1, 2, 1, 0, 1, 0, 0};
    return t[k];
}
__host__ __device__ constexpr int prod_b(int k) {
    constexpr int t[8] = {1, 2, 0, 1, 2, 0, 1, 0};
    return t[k];
}

struct HrArgs {
    float *out;            // output tile base (split 0)
    size_t split_stride;   // elements between split outputs
    int ldo;               // output row pitch (elements)
    int rows;              // valid rows (p)
    int a_plane;           // rows between A planes in the A map (p_pad)
    int b_plane;           // rows between B planes in the B map (d_pad)
    int n_base;            // first H row (output column) of column tile 0
    int n_valid;           // output columns to store, counted from n_base
    int kc_total;          // 64-wide K chunks in d_pad
    int kc_per_split;
    const int *active;     // optional: skip 128-row tiles with no active row
    int *status;
};

template <int BN>
struct HrCfg {
    static constexpr int kTileB = BN * 64 * 2;
    static constexpr int kStage = 3 * kTileA + 3 * kTileB;
    static constexpr int kStages = (200 * 1024) / kStage > 4 ? 4 : (200 * 1024) / kStage;
    static constexpr int kSmem = 1024 + kStages * kStage + 256;
    static constexpr uint32_t kIdesc = tc::idesc_bf16_f32(128, BN);
    static constexpr uint32_t kTmemCols = 4 * BN;  // [buffer][leading, small] accumulators
};

template <int BN>
__global__ void __launch_bounds__(320, 1)
    tc_hr_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                 HrArgs a) {
    using C = HrCfg<BN>;
    constexpr int S = C::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t *bars = (uint64_t *)(smem + S * C::kStage);
    uint32_t *tmem_slot = (uint32_t *)(bars + 2 * S + 4);
    volatile int *abort_flag = (volatile int *)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // tile order: grouped so that consecutive CTAs share column tiles within
    // a band of kGroupRows row tiles (L2 reuse of both operands)
    int tile_m = blockIdx.x, tile_n = blockIdx.y;
    if (gridDim.y > 1) {
        const int lin = blockIdx.y * gridDim.x + blockIdx.x;
        const int per_band = kGroupRows * gridDim.y;
        const int band = lin / per_band, in_band = lin % per_band;
        const int rows_in_band = min(kGroupRows, (int)gridDim.x - band * kGroupRows);
        tile_m = band * kGroupRows + in_band % rows_in_band;
        tile_n = in_band / rows_in_band;
    }
    const int j0 = tile_m * 128;
    const int ncol0 = tile_n * BN;  // relative to n_base
    const int n0 = a.n_base + ncol0;
    const int kc0 = blockIdx.z * a.kc_per_split;
    const int nk = min(a.kc_total, kc0 + a.kc_per_split) - kc0;

    if (a.active) {
        // row activity is written by the scale solve, never by the kernel this
        // launch may overlap, so it can be read before griddepcontrol.wait
        int mine = 0;
        if (threadIdx.x < 128 && j0 + (int)threadIdx.x < a.rows) mine = a.active[j0 + threadIdx.x];
        if (!__syncthreads_or(mine)) {
            tc::pdl_wait();
            return;
        }
    }
    auto full = [&](int s) { return tc::smem_u32(bars + s); };
    auto empty = [&](int s) { return tc::smem_u32(bars + S + s); };
    auto afull = [&](int b) { return tc::smem_u32(bars + 2 * S + b); };
    auto aempty = [&](int b) { return tc::smem_u32(bars + 2 * S + 2 + b); };
    const int nper = nk > 0 ? (nk + kPeriod - 1) / kPeriod : 0;
    auto tileA = [&](int s, int t) { return tc::smem_u32(smem + s * C::kStage + t * kTileA); };
    auto tileB = [&](int s, int t) {
        return tc::smem_u32(smem + s * C::kStage + 3 * kTileA + t * C::kTileB);
    };

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            tc::mbar_init(full(s), 1);
            tc::mbar_init(empty(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            tc::mbar_init(afull(b), 1);
            tc::mbar_init(aempty(b), 8);   // one arrival per drain warp
        }
        *abort_flag = 0;
        tc::fence_barrier_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(tc::smem_u32(tmem_slot), C::kTmemCols);
        tc::tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tc::prefetch_tmap(&mapA);
        tc::prefetch_tmap(&mapB);
    }
    tc::tc_fence_before();
    __syncthreads();
    tc::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // inputs (residual planes) and outputs (partials) are shared with the
    // previous kernel when launched programmatically: wait for it here
    tc::pdl_wait();
    tc::pdl_launch_dependents();

    if (warp == 0 && lane == 0) {
        // ---------------- producer
        int issued = 0;
        for (int c = 0; c < nk; ++c) {
            const int s = c % S;
            const uint32_t ph = (c / S) & 1;
            if (!tc::mbar_wait(empty(s), ph ^ 1) || *abort_flag) {
                *abort_flag = 1;
                break;
            }
            tc::mbar_expect_tx(full(s), C::kStage);
            const int k = (kc0 + c) * 64;
#pragma unroll
            for (int t = 0; t < 3; ++t) tc::tma_load_2d(tileA(s, t), &mapA, full(s), k, j0 + t * a.a_plane);
#pragma unroll
            for (int t = 0; t < 3; ++t) tc::tma_load_2d(tileB(s, t), &mapB, full(s), k, n0 + t * a.b_plane);
            issued = c + 1;
        }
        // copies still in flight complete on their barriers before we leave
        for (int c = issued > S ? issued - S : 0; c < issued; ++c)
            if (!tc::mbar_wait(full(c % S), (c / S) & 1)) *abort_flag = 1;
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        for (int per = 0; per < nper && !*abort_flag; ++per) {
            const int b = per & 1;
            if (!tc::mbar_wait(aempty(b), ((per >> 1) & 1) ^ 1)) {
                *abort_flag = 1;
                break;
            }
            tc::tc_fence_after();
            const uint32_t acc_big = tmem + b * 2 * BN, acc_small = acc_big + BN;
            const int cend = min(nk, (per + 1) * kPeriod);
            for (int c = per * kPeriod; c < cend; ++c) {
                const int s = c % S;
                if (!tc::mbar_wait(full(s), (c / S) & 1) || *abort_flag) {
                    *abort_flag = 1;
                    break;
                }
                tc::tc_fence_after();
                const bool first = (c == per * kPeriod);
#pragma unroll
                for (int sub = 0; sub < 4; ++sub) {
#pragma unroll
                    for (int pr = 0; pr < kProducts; ++pr) {
                        const uint64_t ad = tc::sdesc_sw128(tileA(s, prod_a(pr))) + 2 * sub;
                        const uint64_t bd = tc::sdesc_sw128(tileB(s, prod_b(pr))) + 2 * sub;
                        if (pr == kProducts - 1)
                            tc::mma_bf16(acc_big, ad, bd, C::kIdesc, !(first && sub == 0));
                        else
                            tc::mma_bf16(acc_small, ad, bd, C::kIdesc, !(first && sub == 0 && pr == 0));
                    }
                }
                tc::mma_commit(empty(s));
            }
            tc::mma_commit(afull(b));
        }
    } else if (warp >= 2) {
        // ---------------- drain + store (decisions warp-uniform: tcgen05.ld is .aligned)
        constexpr int HB = BN / 2;                 // columns per drain warp
        const int q = warp & 3, half = (warp - 2) >> 2;
        const int row = j0 + 32 * q + lane;
        float acc[HB];
#pragma unroll
        for (int c = 0; c < HB; ++c) acc[c] = 0.f;
        bool ok = true;
        for (int per = 0; per < nper; ++per) {
            const int b = per & 1;
            bool w = tc::mbar_wait(afull(b), (per >> 1) & 1);
            w = __shfl_sync(0xffffffffu, w && !*abort_flag, 0);
            tc::tc_fence_after();
            if (!w) {
                ok = false;
                *abort_flag = 1;
                break;
            }
            const uint32_t base = tmem + ((uint32_t)(32 * q) << 16) + b * 2 * BN + half * HB;
#pragma unroll
            for (int cc = 0; cc < HB; cc += 16) {
                uint32_t vb[16], vs[16];
                tc::tmem_ld16(base + cc, vb);
                tc::tmem_ld16(base + BN + cc, vs);
                tc::tmem_wait_ld();
#pragma unroll
                for (int e = 0; e < 16; ++e)
                    acc[cc + e] += __uint_as_float(vb[e]) + __uint_as_float(vs[e]);
            }
            tc::tc_fence_before();
            __syncwarp();
            if (lane == 0) tc::mbar_arrive(aempty(b));
        }
        float *orow = a.out + (size_t)blockIdx.z * a.split_stride + (size_t)row * a.ldo;
        if (ok && row < a.rows) {
#pragma unroll
            for (int e = 0; e < HB; e += 4) {
                const int col = ncol0 + half * HB + e;
                if (col + 3 < a.n_valid) {
                    *reinterpret_cast<float4 *>(orow + col) =
                        make_float4(acc[e], acc[e + 1], acc[e + 2], acc[e + 3]);
                } else {
                    for (int u = 0; u < 4; ++u)
                        if (col + u < a.n_valid) orow[col + u] = acc[e + u];
                }
            }
        }
    }
    tc::tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::tc_fence_after();
        tc::tmem_dealloc(tmem, C::kTmemCols);
    }
    if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, ST_TIMEOUT);
}

template <int BN>
cudaError_t launch_tc_hr_bn(const CUtensorMap &mapA, const CUtensorMap &mapB, const HrArgs &a,
                            dim3 grid, cudaStream_t s, bool programmatic = false) {
    using C = HrCfg<BN>;
    static std::atomic<unsigned long long> attr_done{0};
    const cudaError_t e = set_max_dynamic_smem((const void *)tc_hr_kernel<BN>, C::kSmem, attr_done);
    if (e != cudaSuccess) return e;
    if (programmatic) return launch_pdl(tc_hr_kernel<BN>, grid, dim3(320), C::kSmem, s, mapA, mapB, a);
    tc_hr_kernel<BN><<<grid, 320, C::kSmem, s>>>(mapA, mapB, a);
    return cudaGetLastError();
}

}  // namespace

// Full product H r for all rows: out[p][ldo] (columns 0..d-1).
cudaError_t launch_tc_hr_full(const CUtensorMap &mapA, const CUtensorMap &mapB, float *out,
                              int ldo, int p, int p_pad, int d, int d_pad, int *status,
                              cudaStream_t s) {
    HrArgs a{out, 0, ldo, p, p_pad, d_pad, 0, d, d_pad / 64, d_pad / 64, nullptr, status};
    dim3 grid(p_pad / 128, d_pad / 128, 1);
    return launch_tc_hr_bn<128>(mapA, mapB, a, grid, s);
}

// Phase product (H r)_i for group i, split over K: out[split][p][g].
cudaError_t launch_tc_hr_phase(const CUtensorMap &mapA, const CUtensorMap &mapB128,
                               const CUtensorMap &mapB64, float *out, int p, int p_pad, int d_pad,
                               int g, int i, int nsplit, const int *active, int *status,
                               cudaStream_t s) {
    const int kc_total = d_pad / 64;
    const int kc_per = (kc_total + nsplit - 1) / nsplit;
    HrArgs a{out, (size_t)p_pad * g, g, p, p_pad, d_pad, i * g, g, kc_total, kc_per, active, status};
    dim3 grid(p_pad / 128, 1, nsplit);
    if (g == 128) return launch_tc_hr_bn<128>(mapA, mapB128, a, grid, s, true);
    if (g == 64) return launch_tc_hr_bn<64>(mapA, mapB64, a, grid, s, true);
    return cudaErrorInvalidValue;
}

int tc_hr_smem_bytes(int bn) { return bn == 128 ? HrCfg<128>::kSmem : HrCfg<64>::kSmem; }

}  // namespace jarq
