// Objective evaluation without any device allocation.
//
// Some callers cannot allocate device memory at the point where they need
// the objective: serving processes that reserve all device memory up front
// and forbid later cudaMalloc, and callers that must not pay the
// device-wide synchronisation an allocation can imply.  For them
// jarq_objective_noalloc computes the same per-row objective as
// jarq_objective, with every intermediate buffer taken from one statically
// sized device array that exists on each GPU for as long as the library is
// loaded.
//
// The call is synchronous: it waits on the stream twice (after the code
// check and at the end) and reads the handle's status word on the host.
// The array is shared by all calls on a device and keeps the last call's
// contents; the parts that must start at zero (the padding of the bf16
// operand planes) are cleared on every call.  Calls that overlap on the GPU
// (two streams, or two host threads) race on the array.
#include <string.h>

#include "jarq_internal.cuh"

namespace jarq {
namespace {

// Largest padded layer (rows rounded up to 128 times input width rounded up
// to 128) this entry point accepts.
constexpr size_t kNoAllocMaxElems = (size_t)1 << 20;
// r (f32) + residual planes (3 x bf16) + code plane (fp16) + H r (f32), each
// region padded to 256 bytes.
constexpr size_t kRegionR = kNoAllocMaxElems * 4;
constexpr size_t kRegionPlanes = kNoAllocMaxElems * 2 * 3;
constexpr size_t kRegionCodes = kNoAllocMaxElems * 2;
constexpr size_t kRegionHr = kNoAllocMaxElems * 4;
constexpr size_t kScratchBytes = kRegionR + kRegionPlanes + kRegionCodes + kRegionHr;

static __device__ __align__(256) unsigned char g_objective_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
void *g_scratch_ptr[kMaxDevices] = {};

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

bool encode_planes_map(CUtensorMap *m, void *base, uint64_t rows, uint64_t cols) {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) != cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !ptr) {
            (void)cudaGetLastError();
            return false;
        }
        fn = (EncodeTiledFn)ptr;
    }
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {64, 128};
    cuuint32_t es[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

}  // namespace
}  // namespace jarq

using namespace jarq;

extern "C" jarq_status jarq_objective_noalloc(jarq_hessian *h, const float *W, const float *S,
                                              const uint8_t *Q, const int32_t *Z, int dout,
                                              int bits, double *F_per_row, void *stream) {
    if (!h || dout < 0 || bits < 1 || bits > 8) return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    if (!W || !S || !Q || !Z || !F_per_row) return JARQ_ERR_ARG;
    const int d = h->din, d_pad = h->d_pad, g = h->g, G = h->G;
    const int p_pad = round_up(dout, 128);
    if ((size_t)p_pad * (size_t)d_pad > kNoAllocMaxElems) return JARQ_ERR_ARG;
    // the handle's device is current for the call; the caller's is restored
    DeviceGuard dg(h->device);
    if (!dg.ok()) return JARQ_ERR_CUDA;
    // every buffer must already live on this device: staging would allocate
    if (!on_device(W) || !on_device(S) || !on_device(Q) || !on_device(Z) || !on_device(F_per_row))
        return JARQ_ERR_ARG;
    // once per device: the device address of the static scratch array
    if (h->device < 0 || h->device >= kMaxDevices) return JARQ_ERR_ARG;
    if (!g_scratch_ptr[h->device]) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_objective_scratch) != cudaSuccess || !ptr) {
            (void)cudaGetLastError();
            return JARQ_ERR_CUDA;
        }
        g_scratch_ptr[h->device] = ptr;
    }
    unsigned char *base = (unsigned char *)g_scratch_ptr[h->device];
    float *r = (float *)base;
    __nv_bfloat16 *planes = (__nv_bfloat16 *)(base + kRegionR);
    __half *cplane = (__half *)(base + kRegionR + kRegionPlanes);
    float *Hr = (float *)(base + kRegionR + kRegionPlanes + kRegionCodes);
    CUtensorMap mapR;
    if (!encode_planes_map(&mapR, planes, (uint64_t)3 * p_pad, d_pad)) return JARQ_ERR_CUDA;
    cudaStream_t st = (cudaStream_t)stream;
    const ResidualView rv{r, planes, cplane, d, d_pad, p_pad};
    cudaError_t e = cudaMemsetAsync(h->dstatus, 0, sizeof(int), st);
    if (e == cudaSuccess) e = launch_validate(Q, Z, dout, d, G, (1 << bits) - 1, h->dstatus, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->hstatus, h->dstatus, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_CUDA;
    }
    if (*h->hstatus) return JARQ_ERR_ARG;
    // the padding of the operand planes must read as zero
    e = cudaMemsetAsync(planes, 0, (size_t)3 * p_pad * d_pad * 2, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(cplane, 0, (size_t)p_pad * d_pad * 2, st);
    if (e == cudaSuccess) e = launch_residual(W, S, Q, Z, rv, dout, g, st);
    if (e == cudaSuccess)
        e = launch_tc_hr_full(mapR, h->mapH128, Hr, d, dout, p_pad, d, d_pad, h->dstatus, st);
    if (e == cudaSuccess) e = launch_grad(Q, Z, r, Hr, nullptr, F_per_row, dout, d, g, st);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(h->hstatus, h->dstatus, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_CUDA;
    }
    return (*h->hstatus & ST_TIMEOUT) ? JARQ_ERR_TIMEOUT : JARQ_OK;
}
