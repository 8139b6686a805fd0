// Write-back of a refined layer: negative-scale canonicalisation (App. E
// "Representing Negative Scales", Eq. canonicalization), the returned
// weights cast to a weight dtype (Sec. 3.1 Eq. quantized_group; App. E
// "Early stopping"), and b-bit code packing.  The entry points act on device
// memory, allocate nothing and validate the codes first.
#include "jarq_internal.cuh"

namespace jarq {
namespace {

// status word of the write-back calls (device address taken per call)
__device__ int g_writeback_status;

// One warp per (row, group): if s < 0, s' = -s, z' = qmax - z, q' = qmax - q.
__global__ void canonicalize_kernel(float *__restrict__ S, uint8_t *__restrict__ Q,
                                    int32_t *__restrict__ Z, int p, int d, int g, int qmax) {
    const int G = d / g;
    const long long warp = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (warp >= (long long)p * G) return;
    const int j = (int)(warp / G), h = (int)(warp % G);
    const float s = S[(size_t)j * G + h];
    if (!(s < 0.f)) return;   // warp-uniform
    uint8_t *q = Q + (size_t)j * d + (size_t)h * g;
    for (int m = lane; m < g; m += 32) q[m] = (uint8_t)(qmax - q[m]);
    if (lane == 0) {
        S[(size_t)j * G + h] = -s;
        Z[(size_t)j * G + h] = qmax - Z[(size_t)j * G + h];
    }
}

// what = s (q - z): the product of a float32 and an integer of at most 9 bits
// is exact in float64; one rounding to the output type.
template <int DT>
__global__ void dequantize_kernel(const float *__restrict__ S, const uint8_t *__restrict__ Q,
                                  const int32_t *__restrict__ Z, void *__restrict__ out, int p,
                                  int d, int g) {
    const int G = d / g;
    const size_t n = (size_t)p * d;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (size_t)gridDim.x * blockDim.x) {
        const size_t j = idx / d;
        const int grp = (int)(idx - j * d) / g;
        const double w = (double)S[j * G + grp] * (double)((int)Q[idx] - Z[j * G + grp]);
        if (DT == JARQ_F32)
            reinterpret_cast<float *>(out)[idx] = __double2float_rn(w);
        else if (DT == JARQ_F16)
            reinterpret_cast<__half *>(out)[idx] = __double2half(w);
        else
            reinterpret_cast<__nv_bfloat16 *>(out)[idx] = __double2bfloat16(w);
    }
}

// One thread per 32-bit output word: the codes whose bits [k b, k b + b)
// overlap bits [32 w, 32 w + 32) of the row's stream.
__global__ void pack_codes_kernel(const uint8_t *__restrict__ Q, uint32_t *__restrict__ out, int p,
                                  int d, int bits, int nw) {
    const size_t n = (size_t)p * nw;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n;
         idx += (size_t)gridDim.x * blockDim.x) {
        const size_t j = idx / nw;
        const int w = (int)(idx - j * nw);
        const long long lo = 32LL * w, hi = lo + 32;
        const int k0 = (int)(lo / bits), k1 = (int)min((long long)d, (hi + bits - 1) / bits);
        uint64_t v = 0;
        for (int k = k0; k < k1; ++k) {
            const long long pos = (long long)k * bits - lo;   // may be negative for k0
            const uint64_t q = Q[j * d + k];
            v |= pos >= 0 ? (q << pos) : (q >> (-pos));
        }
        out[idx] = (uint32_t)v;
    }
}

int grid_for(size_t n) {
    size_t b = (n + 255) / 256;
    const size_t cap = (size_t)8 * num_sms();
    if (b > cap) b = cap;
    return b < 1 ? 1 : (int)b;
}

// Validate codes (and zero points when Z is given); then run `launch`.
template <class F>
jarq_status checked_run(const uint8_t *Q, const int32_t *Z, int p, int d, int G, int qmax,
                        cudaStream_t st, F launch) {
    int *status = nullptr;
    if (cudaGetSymbolAddress((void **)&status, g_writeback_status) != cudaSuccess || !status) {
        (void)cudaGetLastError();
        return JARQ_ERR_CUDA;
    }
    int host = 0;
    cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int), st);
    if (e == cudaSuccess) e = launch_validate(Q, Z, p, d, Z ? G : 0, qmax, status, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&host, status, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_CUDA;
    }
    if (host) return JARQ_ERR_ARG;
    count_launches(1);
    e = launch(st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_CUDA;
    }
    count_launches(1);
    return JARQ_OK;
}

}  // namespace

bool on_device(const void *p) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    if (at.type == cudaMemoryTypeManaged) return true;
    if (at.type != cudaMemoryTypeDevice) return false;
    int cur = -1;
    if (cudaGetDevice(&cur) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    return at.device == cur;
}

}  // namespace jarq

using namespace jarq;

extern "C" {

jarq_status jarq_canonicalize(float *S, uint8_t *Q, int32_t *Z, int dout, int din, int group_size,
                              int bits, void *stream) {
    if (dout < 0 || din <= 0 || group_size <= 0 || din % group_size || bits < 1 || bits > 8)
        return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    if (!S || !Q || !Z || !on_device(S) || !on_device(Q) || !on_device(Z)) return JARQ_ERR_ARG;
    const int G = din / group_size, qmax = (1 << bits) - 1;
    return checked_run(Q, Z, dout, din, G, qmax, (cudaStream_t)stream, [&](cudaStream_t st) {
        const long long warps = (long long)dout * G;
        canonicalize_kernel<<<(unsigned)((warps * 32 + 255) / 256), 256, 0, st>>>(
            S, Q, Z, dout, din, group_size, qmax);
        return cudaGetLastError();
    });
}

jarq_status jarq_dequantize(const float *S, const uint8_t *Q, const int32_t *Z, int dout, int din,
                            int group_size, int bits, jarq_dtype dtype, void *W_out,
                            void *stream) {
    if (dout < 0 || din <= 0 || group_size <= 0 || din % group_size || bits < 1 || bits > 8 ||
        (dtype != JARQ_F32 && dtype != JARQ_F16 && dtype != JARQ_BF16))
        return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    if (!S || !Q || !Z || !W_out || !on_device(S) || !on_device(Q) || !on_device(Z) ||
        !on_device(W_out))
        return JARQ_ERR_ARG;
    const int G = din / group_size, qmax = (1 << bits) - 1;
    return checked_run(Q, Z, dout, din, G, qmax, (cudaStream_t)stream, [&](cudaStream_t st) {
        const int blocks = grid_for((size_t)dout * din);
        if (dtype == JARQ_F32)
            dequantize_kernel<JARQ_F32><<<blocks, 256, 0, st>>>(S, Q, Z, W_out, dout, din, group_size);
        else if (dtype == JARQ_F16)
            dequantize_kernel<JARQ_F16><<<blocks, 256, 0, st>>>(S, Q, Z, W_out, dout, din, group_size);
        else
            dequantize_kernel<JARQ_BF16><<<blocks, 256, 0, st>>>(S, Q, Z, W_out, dout, din, group_size);
        return cudaGetLastError();
    });
}

jarq_status jarq_pack_codes(const uint8_t *Q, int dout, int din, int bits, uint32_t *packed,
                            void *stream) {
    if (dout < 0 || din <= 0 || bits < 1 || bits > 8) return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    if (!Q || !packed || !on_device(Q) || !on_device(packed)) return JARQ_ERR_ARG;
    const int nw = (int)(((long long)din * bits + 31) / 32);
    return checked_run(Q, nullptr, dout, din, 0, (1 << bits) - 1, (cudaStream_t)stream,
                       [&](cudaStream_t st) {
                           pack_codes_kernel<<<grid_for((size_t)dout * nw), 256, 0, st>>>(
                               Q, packed, dout, din, bits, nw);
                           return cudaGetLastError();
                       });
}

}  // extern "C"
