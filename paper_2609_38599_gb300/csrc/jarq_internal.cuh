// Internal declarations shared by the JARQ CUDA sources (not part of the ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include <atomic>

#include "../../include/jarq.h"

namespace jarq {

// Device status bits (OR-ed by kernels, read back once per call).
enum : int {
    ST_NOT_SPD = 1,      // a diagonal block of H is not positive definite
    ST_NUMERICAL = 2,    // a row's scale system failed even with the ridge
    ST_BAD_CODE = 4,     // a code is outside [0, 2^b - 1]
    ST_BAD_ZERO = 8,     // a zero point is outside [0, 2^b - 1]
    ST_TIMEOUT = 16,     // a bounded device wait gave up
};

constexpr int kMaxGroups = 128;    // largest supported G for the scale solve
constexpr int kSweepSplitTiles = 8;   // row tiles from which the sweep may run as several chains
constexpr int kMaxChains = 4;         // chains of the sweep at most
constexpr int kMaxSplit = 16;      // largest split-K factor of the phase product

__host__ __device__ inline int round_up(int x, int m) { return (x + m - 1) / m * m; }

// View of the residual r = w - D_s (q - z): float32 [p][d] plus its exact
// three-plane bf16 split [3][p_pad][d_pad] read by the tensor cores, and the
// integer codes c = q - z as fp16 [p_pad][d_pad] (exact for |c| <= 2048).
struct ResidualView {
    float *r;
    __nv_bfloat16 *planes;
    __half *cplane;
    int d, d_pad, p_pad;
};

// Exact split x = x1 + x2 + x3 of a float32 into bf16 values (truncation).
__device__ __forceinline__ void split3(float x, __nv_bfloat16 &a, __nv_bfloat16 &b,
                                       __nv_bfloat16 &c) {
    const float x1 = __uint_as_float(__float_as_uint(x) & 0xFFFF0000u);
    const float rem = x - x1;
    const float x2 = __uint_as_float(__float_as_uint(rem) & 0xFFFF0000u);
    a = __float2bfloat16_rz(x1);
    b = __float2bfloat16_rz(x2);
    c = __float2bfloat16_rn(rem - x2);
}

__device__ __forceinline__ void store_code(const ResidualView &v, size_t j, int col, int c) {
    v.cplane[j * v.d_pad + col] = __int2half_rn(c);
}

__device__ __forceinline__ void store_residual(const ResidualView &v, size_t j, int col, float x) {
    v.r[j * v.d + col] = x;
    __nv_bfloat16 a, b, c;
    split3(x, a, b, c);
    const size_t plane = (size_t)v.p_pad * v.d_pad, off = j * v.d_pad + col;
    v.planes[off] = a;
    v.planes[plane + off] = b;
    v.planes[2 * plane + off] = c;
}

// Library-owned refinement workspace, sized for `cap_rows` output rows.
struct Workspace {
    int cap_rows = 0;
    int p_pad = 0;               // rows of the bf16 residual planes (multiple of 128)
    float *Hr = nullptr;         // [p][d]  H r for every row (objective entry point)
    float *r = nullptr;          // [p][d]  residual r = w - D_s (q - z)
    float2 *gram = nullptr;      // [p][G][G]  Gram matrices of the current codes (float pairs)
    double *rhs = nullptr;       // [p][G]  rhs_i = c_i^T P_i (also the scratch of grad)
    float *t_hi = nullptr;       // [nsplit][p_pad][g]  split-K partials of the phase
    float *t_lo = nullptr;       //   product T_i (double-float)
    __nv_bfloat16 *rplanes = nullptr;  // [3][p_pad][d_pad] bf16 split of r
    __half *cplane = nullptr;          // [p_pad][d_pad] codes c = q - z
    CUtensorMap mapR;            // tensor map of rplanes, 128 x 64 boxes
    CUtensorMap mapC;            // tensor map of cplane, 128 x 64 boxes
    // target projection P = W H (once per call); after it the same buffers
    // hold the six digit planes of P for the folded projection
    __nv_bfloat16 *wdig = nullptr;     // [6][p_pad][d_pad] integer digits of W (4) or P (6)
    int *wexp = nullptr;               // [p][G] exponents of those digits
    CUtensorMap mapWd;                 // tensor map of wdig's first 4 planes, 128 x 64 boxes
    CUtensorMap mapPd;                 // tensor map of all 6 planes, 128 x 64 boxes
    float *Phi = nullptr;        // [p][d]  P = Phi + Plo (double-float)
    float *Plo = nullptr;        // [p][d]
    float *Pt_hi = nullptr;      // [p][d]  folded projection Pt_i = R_i^{-T} P_i
    float *Pt_lo = nullptr;      // [p][d]
    double *wHw = nullptr;       // [p]  w_j^T H w_j (||y_j(mu)||^2 for the mu-target)
    double *aux = nullptr;       // [p]  w_j^T XX w_j of the mu-target
    double *own = nullptr;       // [p][G]  c_i^T H_ii w_i (independent scale fit)
    double *L_prev = nullptr;    // [p]  L^{(k-1)} of the early stop
    double *L_host = nullptr;    // [p]
    double *L_final = nullptr;   // [p]
    int *active = nullptr;       // [p]
    int *iters = nullptr;        // [p]
    int *accepted = nullptr;     // [p]
    int *ridge = nullptr;        // [p]
    int *rstat = nullptr;        // [p]
    // staging for host-memory arguments (allocated on first use)
    int stage_rows = 0;
    float *sW = nullptr;
    float *sS = nullptr;
    uint8_t *sQ = nullptr;
    int32_t *sZ = nullptr;
};

}  // namespace jarq

struct jarq_hessian {
    int din = 0, g = 0, G = 0;
    int device = 0;
    int d_pad = 0;
    float *Hs = nullptr;          // [d][d] symmetrised H (+ nu2 I), fp32
    __nv_bfloat16 *Hplanes = nullptr;  // [3][d_pad][d_pad] exact bf16 split of Hs
    // per-block integer digits of Hs (block exponents in expo):
    __nv_bfloat16 *Hdig8 = nullptr;    // [6][d_pad][d_pad] base 2^8, |digit| <= 128
    __half *Hdig10 = nullptr;          // [4][d_pad][d_pad] base 2^10, |digit| <= 512
    int *expo = nullptr;          // [G][G] block exponents of the digits
    CUtensorMap mapH128, mapH64;  // tensor maps of Hplanes, 128 x 64 and 64 x 64 boxes
    CUtensorMap mapD8, mapD10;    // tensor maps of Hdig8 / Hdig10, 64 x 64 boxes
    float *Lf = nullptr;          // [G][g][g] lower factor L_i = R_i^T, row-major
    double *L64 = nullptr;        // [G][g][g] the same in float64
    double *Rinv = nullptr;       // [G][g][g] R_i^{-1} (upper), row-major, float64
    // R_i^{-1} in six base-2^8 digit planes, transposed per block (row i g + a,
    // column b: digit of R_i^{-1}[b][a]), one exponent per group
    __nv_bfloat16 *rdig = nullptr;     // [6][d][g]
    int *rexp = nullptr;               // [G]
    CUtensorMap mapRi;                 // tensor map of rdig, 64 x 64 boxes
    // folded rows Ht[grp i, :] = R_i^{-T} H[grp i, :] in the base-2^10 digit scheme
    __half *Htdig = nullptr;      // [4][d_pad][d_pad] fp16 digits, |digit| <= 512
    int *expoT = nullptr;         // [G][G] block exponents of Ht
    CUtensorMap mapHt;            // tensor map of Htdig, 64 x 64 boxes
    // mu-target (allocated on first use): digits of K or XX, base 2^8, six
    // planes, with a symmetric block-exponent map; staging for host K / XX
    __nv_bfloat16 *qdig = nullptr;     // [6][d_pad][d_pad]
    int *qexp = nullptr;               // [G][G]
    float *qstage = nullptr;           // [d][d]
    CUtensorMap mapQ;                  // tensor map of qdig, 64 x 64 boxes
    int *dstatus = nullptr;       // device status word
    int *hstatus = nullptr;       // pinned host mirror
    // extra streams of the sweep's chains and their fork / join events
    // (made on first use)
    cudaStream_t aux[jarq::kMaxChains - 1] = {};
    cudaEvent_t ev_fork = nullptr, ev_join[jarq::kMaxChains - 1] = {};
    jarq::Workspace ws;
};

namespace jarq {

// ---- launchers (each returns the cudaError_t of its launch) ----
cudaError_t launch_symmetrize(const float *H, float *Hs, __nv_bfloat16 *Hplanes, int d, int d_pad,
                              float nu2, cudaStream_t s);
cudaError_t launch_group_factor(const float *Hs, float *Lf, double *L64, double *Rinv, int d,
                                int g, int *status, cudaStream_t s);
cudaError_t launch_own_rhs(const float *Hs, const float *W, const uint8_t *Q, const int32_t *Z,
                           double *own, int p, int d, int g, cudaStream_t s);
cudaError_t launch_scale_fit(const float2 *gram, const double *rhs, const double *own,
                             const double *wHw, float *S, double *F_before, double *F_after, int p,
                             int G, int method, int passes, cudaStream_t s);
cudaError_t launch_probe(const float *Phi, const float *Plo, const float *t_hi, const float *t_lo,
                         const float *Hs, const double *L64, const float *S, const uint8_t *Q,
                         const int32_t *Z, uint8_t *q_out, int32_t *moves, int32_t *accepted,
                         int32_t *changed, double *dF, int p, int p_pad, int d, int g, int i,
                         int nsplit, int qmax, float eps, cudaStream_t s);
cudaError_t launch_htilde(const float *Hs, const double *Rinv, float *out_hi, float *out_lo,
                          int d, int g, cudaStream_t s);
cudaError_t launch_slice10(const float *hi, const float *lo, int *expo, __half *dig, int d,
                           int d_pad, int g, cudaStream_t s);

cudaError_t launch_validate(const uint8_t *Q, const int32_t *Z, int p, int d, int G, int qmax,
                            int *status, cudaStream_t s);
cudaError_t launch_residual(const float *W, const float *S, const uint8_t *Q, const int32_t *Z,
                            ResidualView rv, int p, int g, cudaStream_t s);
cudaError_t launch_tc_hr_full(const CUtensorMap &mapA, const CUtensorMap &mapB, float *out,
                              int ldo, int p, int p_pad, int d, int d_pad, int *status,
                              cudaStream_t s);
cudaError_t launch_tc_hr_phase(const CUtensorMap &mapA, const CUtensorMap &mapB128,
                               const CUtensorMap &mapB64, float *out, int p, int p_pad, int d_pad,
                               int g, int i, int nsplit, const int *active, int *status,
                               cudaStream_t s);
cudaError_t launch_grad(const uint8_t *Q, const int32_t *Z, const float *r, const float *Hr,
                        double *gvec, double *F, int p, int d, int g, cudaStream_t s);
cudaError_t launch_slices(const float *Hs, int *expo, __nv_bfloat16 *dig8, __half *dig10, int d,
                          int d_pad, int g, cudaStream_t s);
cudaError_t launch_tc_gram(const CUtensorMap &mapC, const CUtensorMap &mapS, const uint8_t *Q,
                           const int32_t *Z, const int *expo, const int *active, float2 *gram,
                           int p, int p_pad, int d, int d_pad, int g, int bits, int *status,
                           cudaStream_t s);
cudaError_t launch_slices8(const float *M, int *expo, __nv_bfloat16 *dig8, int d, int d_pad,
                           int g, cudaStream_t s);
cudaError_t launch_mu_combine(float *Phi, float *Plo, const float *Khi, const float *Klo,
                              const float *W, const double *wXXw, double *wHw, int p, int d,
                              double mu, double nu2, cudaStream_t s);
cudaError_t launch_slice_rows(const float *W, __nv_bfloat16 *planes, int *wexp, int p, int d,
                              int d_pad, int p_pad, int g, cudaStream_t s);
cudaError_t launch_tc_proj(const CUtensorMap &mapW, const CUtensorMap &mapH, float *Phi,
                           float *Plo, const int *wexp, const int *hexp, int p, int p_pad, int d,
                           int d_pad, int g, int *status, cudaStream_t s);
cudaError_t launch_whw(const float *W, const float *Phi, const float *Plo, double *out, int p,
                       int d, cudaStream_t s);
cudaError_t launch_rhs(const uint8_t *Q, const int32_t *Z, const float *Phi, const float *Plo,
                       const int *active, double *rhs, int p, int d, int g, cudaStream_t s);
cudaError_t launch_scale_solve(const float2 *gram, const double *rhs, const double *wHw, float *S,
                               double *L_prev, double *L_out, int *active,
                               int *iters, int *ridge, int *rstat, int *status, int p, int d,
                               int g, int k, bool eval_only, const jarq_options &o,
                               cudaStream_t s);
cudaError_t launch_babai(const float *t_hi, const float *t_lo, const float *pt_hi,
                         const float *pt_lo, int nsplit, const float *Lf, const float *S,
                         uint8_t *Q, const int32_t *Z, ResidualView rv, const int *active,
                         int *accepted, int *status, int p, int g, int i, int qmax, float eps, int row0, int row1,
                         cudaStream_t s, bool pdl = true);
cudaError_t launch_slice_rinv(const double *Rinv, __nv_bfloat16 *rdig, int *rexp, int d, int g,
                              cudaStream_t s);
cudaError_t launch_ptilde(const CUtensorMap &mapPd, const CUtensorMap &mapR, const float *Phi,
                          const float *Plo, __nv_bfloat16 *pdig, int *pexp, const int *rexp,
                          float *out_hi, float *out_lo, int p, int p_pad, int d, int d_pad, int g,
                          int *status, cudaStream_t s);
int target_splits(int p_pad, int g, int G);
cudaError_t launch_wait_timeout(int *status, uint32_t polls, cudaStream_t s);
cudaError_t launch_tc_target(const CUtensorMap &mapC, const CUtensorMap &mapT, float *out_hi,
                             float *out_lo, const float *S, const int *expoT, const int *active,
                             int p, int p_pad, int d_pad, int g, int G, int i, int nsplit,
                             int row0, int nrows, int qmax, int *status, cudaStream_t s,
                             bool pdl = true);

// Launch with programmatic stream serialization: the kernel may start while
// the previous kernel in the stream finishes; it must call griddepcontrol.wait
// before touching that kernel's inputs or outputs.
template <class... KArgs, class... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                     bool pdl, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}
template <class... KArgs, class... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args &&...args) {
    return launch_k(kernel, grid, block, smem, s, true, static_cast<Args &&>(args)...);
}
cudaError_t launch_init_rows(int *active, int *iters, int *accepted, int *ridge, int *rstat,
                             int p, cudaStream_t s);

// Multiprocessor count of the current device (cached per device ordinal).
int num_sms();

// Enable `bytes` of dynamic shared memory for `func` on the current device.
// The attribute is per device and a process may drive several devices, so
// `done` is a bit mask over device ordinals; ordinals of 64 and above set
// the attribute on every call.
cudaError_t set_max_dynamic_smem(const void *func, int bytes,
                                 std::atomic<unsigned long long> &done);

// True for managed memory, or device memory of the current device (a buffer
// on another GPU is false: the kernels would read a peer's memory).
bool on_device(const void *p);

// Makes `device` current for the guard's lifetime and then restores the
// caller's current device, so that an entry point never leaves the calling
// thread on another GPU.
class DeviceGuard {
  public:
    explicit DeviceGuard(int device) {
        if (cudaGetDevice(&prev_) != cudaSuccess) {
            (void)cudaGetLastError();
            return;
        }
        if (prev_ == device) {
            ok_ = true;
            return;
        }
        if (cudaSetDevice(device) == cudaSuccess) {
            ok_ = switched_ = true;
        } else {
            (void)cudaGetLastError();
        }
    }
    ~DeviceGuard() {
        if (switched_) cudaSetDevice(prev_);
    }
    bool ok() const { return ok_; }
    DeviceGuard(const DeviceGuard &) = delete;
    DeviceGuard &operator=(const DeviceGuard &) = delete;

  private:
    int prev_ = 0;
    bool ok_ = false, switched_ = false;
};

// 2D tensor map of 2-byte elements (bf16 or fp16) over [rows][cols]
// (pitch = cols elements), box_rows x 64 boxes, 128-byte swizzle,
// out-of-range elements read as zero.
cudaError_t make_tmap_2b(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols,
                         uint32_t box_rows, CUtensorMapDataType dtype);
cudaError_t make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols,
                           uint32_t box_rows);
cudaError_t make_tmap_f16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols,
                          uint32_t box_rows);

// ---- instrumentation (prof.cu) ----
void count_launches(int n);
void prof_collect();
// Records a CUDA event before construction and, on done(), after the
// launches it brackets, when profiling is enabled.
class ProfScope {
  public:
    ProfScope(const char *name, cudaStream_t s);
    void done();

  private:
    int id_;
    cudaStream_t s_;
    cudaEvent_t a_;
};

}  // namespace jarq
