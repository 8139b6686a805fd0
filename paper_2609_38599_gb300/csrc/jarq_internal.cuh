// Internal declarations shared by the JARQ CUDA sources (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/jarq.h"

namespace jarq {

// Device status bits (OR-ed by kernels, read back once per call).
enum : int {
    ST_NOT_SPD = 1,      // a diagonal block of H is not positive definite
    ST_NUMERICAL = 2,    // a row's scale system failed even with the ridge
    ST_BAD_CODE = 4,     // a code is outside [0, 2^b - 1]
    ST_BAD_ZERO = 8,     // a zero point is outside [0, 2^b - 1]
};

constexpr int kMaxGroup = 128;     // largest supported group size g
constexpr int kMaxGroups = 128;    // largest supported G for the scale solve
constexpr int kSplitK = 4;         // split-K factor of the phase residual product

// Library-owned refinement workspace, sized for `cap_rows` output rows.
struct Workspace {
    int cap_rows = 0;
    float *Hr = nullptr;         // [p][d]  H r for every row (start of an iteration)
    float *r = nullptr;          // [p][d]  residual r = w - D_s (q - z)
    float *gram = nullptr;       // [p][G][G]
    float *gvec = nullptr;       // [p][G]  scale gradient g_i = c_i^T (H r)_i
    float *hr = nullptr;         // [kSplitK][p][g]  split-K partials of (H r)_i
    double *F_start = nullptr;   // [p]  objective at the start of the iteration
    double *L_prev = nullptr;    // [p]  L^{(k-1)} (stop denominator)
    double *dF_sweep = nullptr;  // [p]  sum of accepted Babai dF in the current sweep
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
    float *Hs = nullptr;          // [d][d] symmetrised H (+ nu2 I), fp32
    float *Lf = nullptr;          // [G][g][g] lower factor L_i = R_i^T, row-major
    float *Rinv = nullptr;        // [G][g][g] R_i^{-1} (upper), row-major
    int *dstatus = nullptr;       // device status word
    int *hstatus = nullptr;       // pinned host mirror
    jarq::Workspace ws;
};

namespace jarq {

// ---- launchers (each returns the cudaError_t of its launch) ----
cudaError_t launch_symmetrize(const float *H, float *Hs, int d, float nu2, cudaStream_t s);
cudaError_t launch_group_factor(const float *Hs, float *Lf, float *Rinv, int d, int g,
                                int *status, cudaStream_t s);

cudaError_t launch_validate(const uint8_t *Q, const int32_t *Z, int p, int d, int G, int qmax,
                            int *status, cudaStream_t s);
cudaError_t launch_residual(const float *W, const float *S, const uint8_t *Q, const int32_t *Z,
                            float *r, int p, int d, int g, cudaStream_t s);
cudaError_t launch_hr_full(const float *r, const float *Hs, float *Hr, int p, int d,
                          cudaStream_t s);
cudaError_t launch_grad(const uint8_t *Q, const int32_t *Z, const float *r, const float *Hr,
                        float *gvec, double *F, int p, int d, int g, cudaStream_t s);
cudaError_t launch_gram(const uint8_t *Q, const int32_t *Z, const float *Hs, const int *active,
                        float *gram, int p, int d, int g, cudaStream_t s);
cudaError_t launch_scale_solve(const float *gram, const float *gvec, const float *W,
                               const uint8_t *Q, const int32_t *Z, const double *F_start, float *S,
                               float *r, double *L_prev, double *dF_sweep, int *active,
                               int *iters, int *ridge, int *rstat, int *status, int p, int d,
                               int g, int k, const jarq_options &o, cudaStream_t s);
cudaError_t launch_phase_hr(const float *r, const float *Hs, const int *active, float *hr,
                            int p, int d, int g, int i, cudaStream_t s);
cudaError_t launch_babai(const float *hr, const float *Lf, const float *Rinv, const float *W,
                         const float *S, uint8_t *Q, const int32_t *Z, float *r,
                         const int *active, double *dF_sweep, int *accepted, int p, int d,
                         int g, int i, int qmax, float eps, cudaStream_t s);
cudaError_t launch_init_rows(int *active, int *iters, int *accepted, int *ridge, int *rstat,
                             double *dF_sweep, int p, cudaStream_t s);

int num_sms();

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
