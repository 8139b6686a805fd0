// Double-float arithmetic: pairs (h, l) of float32 with error-free products
// and sums, about 48 significant bits.  GB300 runs float64 at about 1/64 of
// the float32 rate, so the scale solves do no float64 arithmetic in bulk:
// the Gram kernel writes each float64 Gram entry once as such a pair (split
// by integer operations), and the solves work on the pairs.
#pragma once

#include <stdint.h>

namespace jarq {
namespace {

struct DF {
    float h, l;
};

__device__ __forceinline__ DF df_two_sum(float a, float b) {
    const float s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return {s, e};
}

// (h, l) += x * y: the exact product x y = p + pe, p added by two_sum
__device__ __forceinline__ void df_add_prod(DF &a, float x, float y) {
    const float p = __fmul_rn(x, y);
    const float pe = __fmaf_rn(x, y, -p);
    const DF s = df_two_sum(a.h, p);
    a.h = s.h;
    a.l = __fadd_rn(a.l, __fadd_rn(s.l, pe));
}

__device__ __forceinline__ DF df_add(DF a, DF b) {
    const DF s = df_two_sum(a.h, b.h);
    return {s.h, __fadd_rn(s.l, __fadd_rn(a.l, b.l))};
}

__device__ __forceinline__ DF df_neg(DF a) { return {-a.h, -a.l}; }

__device__ __forceinline__ DF df_warp_sum(DF a) {
    // two_sum is exact, so both lanes of a butterfly pair form the same value
    for (int o = 16; o; o >>= 1) {
        const DF b{__shfl_xor_sync(0xffffffffu, a.h, o), __shfl_xor_sync(0xffffffffu, a.l, o)};
        a = df_add(a, b);
    }
    return a;
}

__device__ __forceinline__ double df_to_double(DF a) { return (double)a.h + (double)a.l; }

// x = hi + lo with hi = x rounded to float32 (nearest, ties to even) and
// lo = x - hi rounded to float32, by integer operations on the bits of x.
// Branch-free for zero and for 2^-74 <= |x| < 2^126; any other value
// (tiny, huge, non-finite) sets `rare` and must be split by split_slow.
__device__ __forceinline__ DF split_fast(double x, bool &rare) {
    const unsigned long long bits = (unsigned long long)__double_as_longlong(x);
    const unsigned long long u = bits & 0x7FFFFFFFFFFFFFFFull;
    const int ex = (int)(u >> 52);
    rare = (u != 0) && (ex < 949 || ex > 1148);
    // keep the top 24 significant bits, round to nearest even; a carry out
    // of the mantissa moves into the exponent field, which is still exact
    unsigned long long keep = u >> 29;
    const unsigned long long rem = u & ((1ull << 29) - 1);
    keep += (rem > (1ull << 28)) || (rem == (1ull << 28) && (keep & 1ull));
    // float32 bits: re-bias the exponent from 1023 to 127
    const uint32_t hb = (uint32_t)(keep - (896ull << 23));
    // x - hi in units of x's last place (|r| <= 2^28), times 2^(ex - 1075)
    const int r = (int)(long long)(u - (keep << 29));
    const float unit = __uint_as_float((uint32_t)((ex - 948) & 0xFF) << 23);
    float h = __uint_as_float(hb), l = __fmul_rn(__int2float_rn(r), unit);
    if (u == 0) {
        h = 0.f;
        l = 0.f;
    }
    if (bits >> 63) {
        h = -h;
        l = -l;
    }
    return {h, l};
}

__device__ __noinline__ DF split_slow(double x) {
    const float h = __double2float_rn(x);
    return {h, __double2float_rn(x - (double)h)};
}

__device__ __forceinline__ DF split_double(double x) {
    bool rare;
    const DF v = split_fast(x, rare);
    return rare ? split_slow(x) : v;
}

}  // namespace
}  // namespace jarq
