// Elementwise and bookkeeping kernels of the refinement path.
#include "tc_common.cuh"

namespace jarq {
namespace {

// Codes and zero points must lie in [0, qmax] (Sec. 3.1: q in B^{d_i};
// integer zero points kept from the host).
__global__ void validate_kernel(const uint8_t *__restrict__ Q, const int32_t *__restrict__ Z,
                                size_t nq, size_t nz, int qmax, int *status) {
    __shared__ int flag;
    if (threadIdx.x == 0) flag = 0;
    __syncthreads();
    int local = 0;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nq; i += stride)
        if (Q[i] > qmax) local |= ST_BAD_CODE;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nz; i += stride)
        if (Z[i] < 0 || Z[i] > qmax) local |= ST_BAD_ZERO;
    if (local) atomicOr(&flag, local);
    __syncthreads();
    if (threadIdx.x == 0 && flag) atomicOr(status, flag);
}

// The same check, sixteen codes per thread (Q 16-byte aligned, nq a
// multiple of 16).
__global__ void validate16_kernel(const uint4 *__restrict__ Q16, const int32_t *__restrict__ Z,
                                  size_t nq16, size_t nz, int qmax, int *status) {
    __shared__ int flag;
    if (threadIdx.x == 0) flag = 0;
    __syncthreads();
    int local = 0;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nq16; i += stride) {
        const uint4 v = Q16[i];
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
            for (int b = 0; b < 4; ++b)
                if ((int)((w4[k] >> (8 * b)) & 0xFFu) > qmax) local |= ST_BAD_CODE;
    }
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < nz; i += stride)
        if (Z[i] < 0 || Z[i] > qmax) local |= ST_BAD_ZERO;
    if (local) atomicOr(&flag, local);
    __syncthreads();
    if (threadIdx.x == 0 && flag) atomicOr(status, flag);
}

// r = w - s (q - z), one rounding (fma) per element (Eq. quantized_group),
// and the code plane c = q - z; with rv.r == nullptr only the code plane.
__global__ void residual_kernel(const float *__restrict__ W, const float *__restrict__ S,
                                const uint8_t *__restrict__ Q, const int32_t *__restrict__ Z,
                                ResidualView rv, int p, int g) {
    const int d = rv.d, G = d / g;
    const size_t n = (size_t)p * d;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    for (size_t idx = (size_t)blockIdx.x * blockDim.x + threadIdx.x; idx < n; idx += stride) {
        const size_t j = idx / d;
        const int grp = (int)(idx - j * d) / g;
        const int ci = (int)Q[idx] - Z[j * G + grp];
        if (rv.r) store_residual(rv, j, (int)(idx - j * d), fmaf(-S[j * G + grp], (float)ci, W[idx]));
        store_code(rv, j, (int)(idx - j * d), ci);
    }
}

// Only the code plane c = q - z, eight codes per thread (one group: g is a
// multiple of 8; Q 8-byte aligned; 16-byte stores into the plane).
__global__ void codes_kernel(const uint8_t *__restrict__ Q, const int32_t *__restrict__ Z,
                             ResidualView rv, int p, int g) {
    const int d = rv.d, G = d / g;
    const size_t n8 = (size_t)p * d / 8;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    for (size_t i8 = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i8 < n8; i8 += stride) {
        const size_t idx = i8 * 8;
        const size_t j = idx / d;
        const int col = (int)(idx - j * d);
        const int z = Z[j * G + col / g];
        const uint2 q8 = *reinterpret_cast<const uint2 *>(Q + idx);
        const uint32_t w2[2] = {q8.x, q8.y};
        __align__(16) __half h[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) h[k] = __int2half_rn((int)((w2[k >> 2] >> (8 * (k & 3))) & 0xFFu) - z);
        *reinterpret_cast<uint4 *>(rv.cplane + j * rv.d_pad + col) = *reinterpret_cast<const uint4 *>(h);
    }
}

__global__ void init_rows_kernel(int *active, int *iters, int *accepted, int *ridge, int *rstat,
                                 int p) {
    int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j < p) {
        active[j] = 1;
        iters[j] = 0;
        accepted[j] = 0;
        ridge[j] = 0;
        rstat[j] = 0;
    }
}

}  // namespace

int num_sms() {
    constexpr int kDevs = 64;
    static std::atomic<int> cache[kDevs];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        dev = 0;
    }
    const bool cached = dev >= 0 && dev < kDevs;
    int n = cached ? cache[dev].load(std::memory_order_relaxed) : 0;
    if (n > 0) return n;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
        (void)cudaGetLastError();
        n = 0;
    }
    if (n <= 0) n = 1;
    if (cached) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

cudaError_t set_max_dynamic_smem(const void *func, int bytes,
                                 std::atomic<unsigned long long> &done) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = (dev >= 0 && dev < 64) ? (1ull << dev) : 0ull;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_acq_rel);
    return e;
}

cudaError_t launch_validate(const uint8_t *Q, const int32_t *Z, int p, int d, int G, int qmax,
                            int *status, cudaStream_t s) {
    size_t nq = (size_t)p * d, nz = (size_t)p * G;
    int blocks = (int)((nq + 255) / 256);
    if (blocks > 4 * num_sms()) blocks = 4 * num_sms();
    if (blocks < 1) blocks = 1;
    if (nq % 16 == 0 && (uintptr_t)Q % 16 == 0)
        validate16_kernel<<<blocks, 256, 0, s>>>(reinterpret_cast<const uint4 *>(Q), Z, nq / 16, nz,
                                                 qmax, status);
    else
        validate_kernel<<<blocks, 256, 0, s>>>(Q, Z, nq, nz, qmax, status);
    return cudaGetLastError();
}

cudaError_t launch_residual(const float *W, const float *S, const uint8_t *Q, const int32_t *Z,
                            ResidualView rv, int p, int g, cudaStream_t s) {
    size_t n = (size_t)p * rv.d;
    int blocks = (int)((n + 255) / 256);
    if (blocks > 8 * num_sms()) blocks = 8 * num_sms();
    if (blocks < 1) blocks = 1;
    if (!rv.r && g % 8 == 0 && (uintptr_t)Q % 8 == 0 && rv.d_pad % 8 == 0)
        codes_kernel<<<blocks, 256, 0, s>>>(Q, Z, rv, p, g);
    else
        residual_kernel<<<blocks, 256, 0, s>>>(W, S, Q, Z, rv, p, g);
    return cudaGetLastError();
}

cudaError_t launch_init_rows(int *active, int *iters, int *accepted, int *ridge, int *rstat,
                             int p, cudaStream_t s) {
    init_rows_kernel<<<(p + 255) / 256, 256, 0, s>>>(active, iters, accepted, ridge, rstat, p);
    return cudaGetLastError();
}

// A wait that nothing completes: one thread polls a fresh mbarrier (count 1,
// no arrival), gives up after `polls` polls and records ST_TIMEOUT, as every
// kernel of the library does when one of its bounded waits runs out.
__global__ void wait_timeout_kernel(int *status, uint32_t polls) {
    __shared__ uint64_t bar;
    if (threadIdx.x != 0) return;
    const uint32_t b = tc::smem_u32(&bar);
    tc::mbar_init(b, 1);
    tc::fence_barrier_init();
    bool done = false;
    for (uint32_t i = 0; i < polls && !done; ++i) done = tc::mbar_try_wait(b, 0);
    if (!done) atomicOr(status, ST_TIMEOUT);
}

cudaError_t launch_wait_timeout(int *status, uint32_t polls, cudaStream_t s) {
    wait_timeout_kernel<<<1, 32, 0, s>>>(status, polls);
    return cudaGetLastError();
}

}  // namespace jarq
