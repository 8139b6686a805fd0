// C ABI entry points: handle lifecycle, argument checks, staging of host
// buffers and the refinement loop (Sec. 3.3; App. E "Order of updates").
//
// Once per call: the target projection P = W H, w^T H w and the folded
// projection Pt_i = R_i^{-T} P_i (App. G "Computational Complexity",
// target-projection shortcut).  Per iteration k = 1..K: the Gram matrices of
// the current codes and rhs_i = c_i^T P_i, the joint scale solve (gradient
// rhs - Gram s, objective, early stop), and one Gauss-Seidel sweep over the
// groups, each group being a target-product phase (T_i) followed by a Babai
// phase on y = (Pt_i - T_i) / s_i.
#include <float.h>
#include <stdlib.h>
#include <string.h>

#include <new>

#include "jarq_internal.cuh"

namespace jarq {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// 2D tensor map of 2-byte elements (bf16 or fp16) over [rows][cols]
// (pitch = cols), box_rows x 64 boxes, 128-byte swizzle, out-of-range
// elements read as zero.
cudaError_t make_tmap_2b(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols,
                         uint32_t box_rows, CUtensorMapDataType dtype) {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                                         cudaEnableDefault, &q);
        if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !ptr)
            return e != cudaSuccess ? e : cudaErrorSymbolNotFound;
        fn = (EncodeTiledFn)ptr;
    }
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t es[2] = {1, 1};
    CUresult r = fn(m, dtype, 2, const_cast<void *>(base), dims, strides,
                    box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

cudaError_t make_tmap_bf16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols,
                           uint32_t box_rows) {
    return make_tmap_2b(m, base, rows, cols, box_rows, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16);
}

cudaError_t make_tmap_f16(CUtensorMap *m, const void *base, uint64_t rows, uint64_t cols,
                          uint32_t box_rows) {
    return make_tmap_2b(m, base, rows, cols, box_rows, CU_TENSOR_MAP_DATA_TYPE_FLOAT16);
}

}  // namespace jarq

using namespace jarq;

namespace {

jarq_status cuda_fail(cudaError_t e) {
    return e == cudaErrorMemoryAllocation ? JARQ_ERR_NOMEM : JARQ_ERR_CUDA;
}

#define CK(x)                                  \
    do {                                       \
        cudaError_t e_ = (x);                  \
        if (e_ != cudaSuccess) {               \
            (void)cudaGetLastError();          \
            return cuda_fail(e_);              \
        }                                      \
    } while (0)

// Launch `call` (which enqueues `n` kernels on stream `strm`) under the
// profiling scope `name`.
#define RUN_ON(name, n, strm, call)     \
    do {                                \
        ProfScope ps_(name, strm);      \
        CK(call);                       \
        ps_.done();                     \
        count_launches(n);              \
    } while (0)
#define RUN(name, n, call) RUN_ON(name, n, st, call)

template <class T>
cudaError_t dalloc(T **p, size_t n) {
    *p = nullptr;
    if (n == 0) n = 1;
    return cudaMalloc((void **)p, n * sizeof(T));
}

bool is_device_ptr(const void *ptr) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, ptr) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged;
}

void free_ws(Workspace &w) {
    cudaFree(w.Hr);
    cudaFree(w.r);
    cudaFree(w.gram);
    cudaFree(w.rhs);
    cudaFree(w.t_hi);
    cudaFree(w.t_lo);
    cudaFree(w.Pt_hi);
    cudaFree(w.Pt_lo);
    cudaFree(w.wdig);
    cudaFree(w.wexp);
    cudaFree(w.Phi);
    cudaFree(w.Plo);
    cudaFree(w.wHw);
    cudaFree(w.aux);
    cudaFree(w.own);
    cudaFree(w.L_prev);
    cudaFree(w.L_host);
    cudaFree(w.L_final);
    cudaFree(w.active);
    cudaFree(w.iters);
    cudaFree(w.accepted);
    cudaFree(w.ridge);
    cudaFree(w.rstat);
    cudaFree(w.sW);
    cudaFree(w.sS);
    cudaFree(w.sQ);
    cudaFree(w.sZ);
    cudaFree(w.rplanes);
    cudaFree(w.cplane);
    w = Workspace{};
}

cudaError_t ensure_ws(jarq_hessian *h, int p) {
    Workspace &w = h->ws;
    if (p <= w.cap_rows) return cudaSuccess;
    free_ws(w);
    const size_t d = h->din, G = h->G, g = h->g;
    const int p_pad = round_up(p, 128);
    cudaError_t e;
    if ((e = dalloc(&w.rplanes, (size_t)3 * p_pad * h->d_pad)) != cudaSuccess) return e;
    if ((e = cudaMemset(w.rplanes, 0, (size_t)3 * p_pad * h->d_pad * 2)) != cudaSuccess) return e;
    if ((e = make_tmap_bf16(&w.mapR, w.rplanes, (uint64_t)3 * p_pad, h->d_pad, 128)) != cudaSuccess)
        return e;
    if ((e = dalloc(&w.cplane, (size_t)p_pad * h->d_pad)) != cudaSuccess) return e;
    if ((e = cudaMemset(w.cplane, 0, (size_t)p_pad * h->d_pad * 2)) != cudaSuccess) return e;
    if ((e = make_tmap_f16(&w.mapC, w.cplane, (uint64_t)p_pad, h->d_pad, 128)) != cudaSuccess)
        return e;
    if ((e = dalloc(&w.wdig, (size_t)6 * p_pad * h->d_pad)) != cudaSuccess) return e;
    if ((e = cudaMemset(w.wdig, 0, (size_t)6 * p_pad * h->d_pad * 2)) != cudaSuccess) return e;
    if ((e = make_tmap_bf16(&w.mapWd, w.wdig, (uint64_t)4 * p_pad, h->d_pad, 128)) != cudaSuccess)
        return e;
    if ((e = make_tmap_bf16(&w.mapPd, w.wdig, (uint64_t)6 * p_pad, h->d_pad, 128)) != cudaSuccess)
        return e;
    w.p_pad = p_pad;
    if ((e = dalloc(&w.Hr, (size_t)p * d)) != cudaSuccess) return e;
    if ((e = dalloc(&w.r, (size_t)p * d)) != cudaSuccess) return e;
    if ((e = dalloc(&w.gram, (size_t)p * G * G)) != cudaSuccess) return e;
    if ((e = dalloc(&w.rhs, (size_t)p * G)) != cudaSuccess) return e;
    if ((e = dalloc(&w.t_hi, (size_t)kMaxSplit * p_pad * g)) != cudaSuccess) return e;
    if ((e = dalloc(&w.t_lo, (size_t)kMaxSplit * p_pad * g)) != cudaSuccess) return e;
    if ((e = dalloc(&w.Pt_hi, (size_t)p * d)) != cudaSuccess) return e;
    if ((e = dalloc(&w.Pt_lo, (size_t)p * d)) != cudaSuccess) return e;
    if ((e = dalloc(&w.wexp, (size_t)p * G)) != cudaSuccess) return e;
    if ((e = dalloc(&w.Phi, (size_t)p * d)) != cudaSuccess) return e;
    if ((e = dalloc(&w.Plo, (size_t)p * d)) != cudaSuccess) return e;
    if ((e = dalloc(&w.wHw, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.aux, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.own, (size_t)p * G)) != cudaSuccess) return e;
    if ((e = dalloc(&w.L_prev, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.L_host, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.L_final, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.active, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.iters, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.accepted, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.ridge, (size_t)p)) != cudaSuccess) return e;
    if ((e = dalloc(&w.rstat, (size_t)p)) != cudaSuccess) return e;
    w.cap_rows = p;
    return cudaSuccess;
}

// Joins the first n extra streams of the sweep to `st` when it goes out of
// scope: an error return in the middle of a sweep leaves no work of this
// call running unordered with the caller's stream (best effort: the errors
// of the join itself are dropped).
struct ChainJoin {
    jarq_hessian *h;
    cudaStream_t st;
    int n;
    ~ChainJoin() {
        if (n == 0) return;
        for (int c = 0; c < n; ++c)
            if (cudaEventRecord(h->ev_join[c], h->aux[c]) == cudaSuccess)
                (void)cudaStreamWaitEvent(st, h->ev_join[c], 0);
        (void)cudaGetLastError();
    }
};

// Device views of the four layer arguments, staging host buffers.
struct LayerArgs {
    const float *W;
    float *S;
    uint8_t *Q;
    const int32_t *Z;
    bool hS = false, hQ = false;  // S / Q came from host memory
};

cudaError_t stage_layer(jarq_hessian *h, const float *W, const float *S, const uint8_t *Q,
                        const int32_t *Z, int p, LayerArgs &out, cudaStream_t st) {
    Workspace &w = h->ws;
    const size_t d = h->din, G = h->G;
    // the kernels read the codes in 16-byte vectors: a device Q that is not
    // 16-byte aligned is staged like host memory
    const bool dW = is_device_ptr(W), dS = is_device_ptr(S),
               dQ = is_device_ptr(Q) && ((uintptr_t)Q & 15) == 0, dZ = is_device_ptr(Z);
    if ((!dW || !dS || !dQ || !dZ) && w.stage_rows < p) {
        cudaFree(w.sW);
        cudaFree(w.sS);
        cudaFree(w.sQ);
        cudaFree(w.sZ);
        w.sW = nullptr;
        w.sS = nullptr;
        w.sQ = nullptr;
        w.sZ = nullptr;
        w.stage_rows = 0;
        cudaError_t e;
        if ((e = dalloc(&w.sW, (size_t)p * d)) != cudaSuccess) return e;
        if ((e = dalloc(&w.sS, (size_t)p * G)) != cudaSuccess) return e;
        if ((e = dalloc(&w.sQ, (size_t)p * d)) != cudaSuccess) return e;
        if ((e = dalloc(&w.sZ, (size_t)p * G)) != cudaSuccess) return e;
        w.stage_rows = p;
    }
    out.W = W;
    out.S = const_cast<float *>(S);
    out.Q = const_cast<uint8_t *>(Q);
    out.Z = Z;
    cudaError_t e = cudaSuccess;
    if (!dW) {
        e = cudaMemcpyAsync(w.sW, W, (size_t)p * d * sizeof(float), cudaMemcpyHostToDevice, st);
        out.W = w.sW;
    }
    if (e == cudaSuccess && !dS) {
        e = cudaMemcpyAsync(w.sS, S, (size_t)p * G * sizeof(float), cudaMemcpyHostToDevice, st);
        out.S = w.sS;
        out.hS = true;
    }
    if (e == cudaSuccess && !dQ) {
        e = cudaMemcpyAsync(w.sQ, Q, (size_t)p * d, cudaMemcpyDefault, st);
        out.Q = w.sQ;
        out.hQ = true;
    }
    if (e == cudaSuccess && !dZ) {
        e = cudaMemcpyAsync(w.sZ, Z, (size_t)p * G * sizeof(int32_t), cudaMemcpyHostToDevice,
                            st);
        out.Z = w.sZ;
    }
    return e;
}

jarq_status status_from_bits(int bits) {
    if (bits & ST_NOT_SPD) return JARQ_ERR_NOT_SPD;
    if (bits & (ST_BAD_CODE | ST_BAD_ZERO)) return JARQ_ERR_ARG;
    if (bits & ST_TIMEOUT) return JARQ_ERR_TIMEOUT;
    if (bits & ST_NUMERICAL) return JARQ_ERR_NUMERICAL;
    return JARQ_OK;
}

cudaError_t read_status(jarq_hessian *h, cudaStream_t st, int *bits) {
    cudaError_t e = cudaMemcpyAsync(h->hstatus, h->dstatus, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    *bits = (e == cudaSuccess) ? *h->hstatus : 0;
    if (e == cudaSuccess) prof_collect();
    return e;
}

ResidualView rview(jarq_hessian *h) {
    return ResidualView{h->ws.r, h->ws.rplanes, h->ws.cplane, h->din, h->d_pad, h->ws.p_pad};
}

// Common front half of refine/objective: stage, validate, residual.
jarq_status layer_front(jarq_hessian *h, const float *W, const float *S, const uint8_t *Q,
                        const int32_t *Z, int dout, int bits, LayerArgs &la, cudaStream_t st,
                        bool codes_only = false) {
    CK(cudaSetDevice(h->device));
    CK(ensure_ws(h, dout));
    CK(stage_layer(h, W, S, Q, Z, dout, la, st));
    CK(cudaMemsetAsync(h->dstatus, 0, sizeof(int), st));
    RUN("validate", 1, launch_validate(la.Q, la.Z, dout, h->din, h->G, (1 << bits) - 1, h->dstatus, st));
    int sb = 0;
    CK(read_status(h, st, &sb));
    if (sb) return status_from_bits(sb);
    ResidualView rv = rview(h);
    if (codes_only) rv.r = nullptr;
    RUN("residual", 1, launch_residual(la.W, la.S, la.Q, la.Z, rv, dout, h->g, st));
    return JARQ_OK;
}

bool layer_args_ok(const jarq_hessian *h, const void *W, const void *S, const void *Q,
                   const void *Z, int dout, int bits) {
    if (!h || dout < 0 || bits < 1 || bits > 8) return false;
    if (dout > 0 && (!W || !S || !Q || !Z)) return false;
    return true;
}

// Inputs of the propagation-corrected target (App. "Propagation-Corrected
// Targets and QEP"): K = X~^T X and XX = X^T X, float32 [d][d] with the
// normalisation of the prepared H, and mu, nu^2.
struct MuTarget {
    const float *K, *XX;
    float mu, nu2;
};

jarq_status refine_impl(jarq_hessian *h, const float *W, float *S, uint8_t *Q, const int32_t *Z,
                        int dout, int bits, const jarq_options *opt, jarq_stats *stats,
                        void *stream, const MuTarget *mt);

// Digits of a d x d float32 matrix M (host or device) into the handle's
// mu-target planes, then its target projection W M^T into (out_hi, out_lo).
jarq_status project_by(jarq_hessian *h, const float *M, int p, float *out_hi, float *out_lo,
                       cudaStream_t st) {
    Workspace &w = h->ws;
    const int d = h->din, g = h->g;
    if (!h->qdig) {
        CK(dalloc(&h->qdig, (size_t)6 * h->d_pad * h->d_pad));
        CK(cudaMemset(h->qdig, 0, (size_t)6 * h->d_pad * h->d_pad * 2));
        CK(dalloc(&h->qexp, (size_t)h->G * h->G));
        CK(make_tmap_bf16(&h->mapQ, h->qdig, (uint64_t)6 * h->d_pad, h->d_pad, 64));
    }
    const float *Md = M;
    if (!is_device_ptr(M)) {
        if (!h->qstage) CK(dalloc(&h->qstage, (size_t)d * d));
        CK(cudaMemcpyAsync(h->qstage, M, (size_t)d * d * sizeof(float), cudaMemcpyHostToDevice, st));
        Md = h->qstage;
    }
    RUN("slices", 2, launch_slices8(Md, h->qexp, h->qdig, d, h->d_pad, g, st));
    RUN("proj", 1, launch_tc_proj(w.mapWd, h->mapQ, out_hi, out_lo, w.wexp, h->qexp, p, w.p_pad,
                                  d, h->d_pad, g, h->dstatus, st));
    return JARQ_OK;
}

// H w_corr and ||y(mu)||^2 in place of H w and w^T H w (Eqs. mu-target,
// w-corr): w^T XX w from the projection by XX, then the projection by K
// and the combination.
jarq_status mu_projection(jarq_hessian *h, const float *Wd, int p, const MuTarget &t,
                          cudaStream_t st) {
    Workspace &w = h->ws;
    const int d = h->din;
    jarq_status rc = project_by(h, t.XX, p, w.Pt_hi, w.Pt_lo, st);
    if (rc != JARQ_OK) return rc;
    RUN("whw", 1, launch_whw(Wd, w.Pt_hi, w.Pt_lo, w.aux, p, d, st));
    rc = project_by(h, t.K, p, w.Pt_hi, w.Pt_lo, st);
    if (rc != JARQ_OK) return rc;
    RUN("mu_combine", 1, launch_mu_combine(w.Phi, w.Plo, w.Pt_hi, w.Pt_lo, Wd, w.aux, w.wHw, p, d,
                                           (double)t.mu, (double)t.nu2, st));
    return JARQ_OK;
}

}  // namespace

extern "C" {

jarq_options jarq_default_options(void) {
    jarq_options o;
    o.max_iters = 3;
    o.early_stop = 1;
    o.tau_rel = 1e-5f;
    o.tau_abs = 1e-5f;
    o.ridge = 1e-4f;
    o.rcond = 1e-10f;
    o.eps = FLT_EPSILON;
    o.ridge_accept = 0;
    o.fixed_grid = 0;
    return o;
}

jarq_status jarq_selftest_wait_timeout(void *stream) {
    cudaStream_t st = (cudaStream_t)stream;
    int *d = nullptr;
    int bits = 0;
    if (cudaMalloc(&d, sizeof(int)) != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_NOMEM;
    }
    cudaError_t e = cudaMemsetAsync(d, 0, sizeof(int), st);
    if (e == cudaSuccess) e = launch_wait_timeout(d, 256, st);
    if (e == cudaSuccess) e = cudaMemcpyAsync(&bits, d, sizeof(int), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    cudaFree(d);
    if (e != cudaSuccess) {
        (void)cudaGetLastError();
        return JARQ_ERR_CUDA;
    }
    return status_from_bits(bits);
}

const char *jarq_status_string(jarq_status s) {
    switch (s) {
        case JARQ_OK: return "ok";
        case JARQ_ERR_ARG: return "invalid argument";
        case JARQ_ERR_NOT_SPD: return "Hessian diagonal block not positive definite";
        case JARQ_ERR_NUMERICAL: return "scale system failed even with the ridge";
        case JARQ_ERR_CUDA: return "CUDA error";
        case JARQ_ERR_TIMEOUT: return "device wait timed out";
        case JARQ_ERR_NOMEM: return "device allocation failed";
    }
    return "unknown status";
}

int jarq_hessian_din(const jarq_hessian *h) { return h ? h->din : 0; }
int jarq_hessian_group_size(const jarq_hessian *h) { return h ? h->g : 0; }

void jarq_hessian_destroy(jarq_hessian *h) {
    if (!h) return;
    DeviceGuard dg(h->device);
    cudaDeviceSynchronize();
    free_ws(h->ws);
    cudaFree(h->Hs);
    cudaFree(h->Hplanes);
    cudaFree(h->Hdig8);
    cudaFree(h->Hdig10);
    cudaFree(h->expo);
    cudaFree(h->Lf);
    cudaFree(h->L64);
    cudaFree(h->Rinv);
    cudaFree(h->rdig);
    cudaFree(h->rexp);
    cudaFree(h->Htdig);
    cudaFree(h->expoT);
    cudaFree(h->qdig);
    cudaFree(h->qexp);
    cudaFree(h->qstage);
    cudaFree(h->dstatus);
    cudaFreeHost(h->hstatus);
    if (h->ev_fork) cudaEventDestroy(h->ev_fork);
    for (int c = 0; c < kMaxChains - 1; ++c) {
        if (h->ev_join[c]) cudaEventDestroy(h->ev_join[c]);
        if (h->aux[c]) cudaStreamDestroy(h->aux[c]);
    }
    (void)cudaGetLastError();
    delete h;
}

jarq_status jarq_prepare_hessian(const float *H, int din, int group_size, float nu2,
                                 jarq_hessian **out, void *stream) {
    if (!H || !out || din <= 0 || (group_size != 64 && group_size != 128) ||
        din % group_size != 0 || din / group_size > kMaxGroups || !isfinite(nu2))
        return JARQ_ERR_ARG;
    cudaStream_t st = (cudaStream_t)stream;
    jarq_hessian *h = new (std::nothrow) jarq_hessian();
    if (!h) return JARQ_ERR_NOMEM;
    h->din = din;
    h->g = group_size;
    h->G = din / group_size;
    h->d_pad = round_up(din, 128);
    jarq_status rc = JARQ_OK;
    float *Hdev = nullptr, *Ht_hi = nullptr, *Ht_lo = nullptr;
    do {
        if (cudaGetDevice(&h->device) != cudaSuccess) { rc = JARQ_ERR_CUDA; break; }
        const size_t dd = (size_t)din * din;
        cudaError_t e;
        if ((e = dalloc(&h->Hs, dd)) != cudaSuccess) { rc = cuda_fail(e); break; }
        const size_t pd = (size_t)h->d_pad * h->d_pad;
        if ((e = dalloc(&h->Hplanes, 3 * pd)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = cudaMemsetAsync(h->Hplanes, 0, 3 * pd * 2, st)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = make_tmap_bf16(&h->mapH128, h->Hplanes, (uint64_t)3 * h->d_pad, h->d_pad, 128)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = make_tmap_bf16(&h->mapH64, h->Hplanes, (uint64_t)3 * h->d_pad, h->d_pad, 64)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->Hdig8, 6 * pd)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = cudaMemsetAsync(h->Hdig8, 0, 6 * pd * 2, st)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->Hdig10, 4 * pd)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = cudaMemsetAsync(h->Hdig10, 0, 4 * pd * 2, st)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->expo, (size_t)h->G * h->G)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = make_tmap_bf16(&h->mapD8, h->Hdig8, (uint64_t)6 * h->d_pad, h->d_pad, 64)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = make_tmap_f16(&h->mapD10, h->Hdig10, (uint64_t)4 * h->d_pad, h->d_pad, 64)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->Lf, (size_t)h->G * group_size * group_size)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->L64, (size_t)h->G * group_size * group_size)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->Rinv, (size_t)h->G * group_size * group_size)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->rdig, (size_t)6 * din * group_size)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->rexp, (size_t)h->G)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = make_tmap_bf16(&h->mapRi, h->rdig, (uint64_t)6 * din, group_size, 64)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->Htdig, 4 * pd)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = cudaMemsetAsync(h->Htdig, 0, 4 * pd * 2, st)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->expoT, (size_t)h->G * h->G)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = make_tmap_f16(&h->mapHt, h->Htdig, (uint64_t)4 * h->d_pad, h->d_pad, 64)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&h->dstatus, 1)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = cudaMallocHost((void **)&h->hstatus, sizeof(int))) != cudaSuccess) { rc = cuda_fail(e); break; }
        const float *Hsrc = H;
        if (!is_device_ptr(H)) {
            if ((e = dalloc(&Hdev, dd)) != cudaSuccess) { rc = cuda_fail(e); break; }
            if ((e = cudaMemcpyAsync(Hdev, H, dd * sizeof(float), cudaMemcpyHostToDevice, st)) != cudaSuccess) { rc = cuda_fail(e); break; }
            Hsrc = Hdev;
        }
        if ((e = cudaMemsetAsync(h->dstatus, 0, sizeof(int), st)) != cudaSuccess) { rc = cuda_fail(e); break; }
        { ProfScope ps("symmetrize", st); e = launch_symmetrize(Hsrc, h->Hs, h->Hplanes, din, h->d_pad, nu2, st); ps.done(); count_launches(1); }
        if (e != cudaSuccess) { rc = cuda_fail(e); break; }
        { ProfScope ps("group_factor", st); e = launch_group_factor(h->Hs, h->Lf, h->L64, h->Rinv, din, group_size, h->dstatus, st); ps.done(); count_launches(1); }
        if (e != cudaSuccess) { rc = cuda_fail(e); break; }
        { ProfScope ps("slices", st); e = launch_slice_rinv(h->Rinv, h->rdig, h->rexp, din, group_size, st); ps.done(); count_launches(1); }
        if (e != cudaSuccess) { rc = cuda_fail(e); break; }
        // folded rows R_i^{-T} H[grp i, :] (double-float, temporary) -> digits
        if ((e = dalloc(&Ht_hi, dd)) != cudaSuccess) { rc = cuda_fail(e); break; }
        if ((e = dalloc(&Ht_lo, dd)) != cudaSuccess) { rc = cuda_fail(e); break; }
        { ProfScope ps("htilde", st); e = launch_htilde(h->Hs, h->Rinv, Ht_hi, Ht_lo, din, group_size, st); ps.done(); count_launches(1); }
        if (e != cudaSuccess) { rc = cuda_fail(e); break; }
        { ProfScope ps("slices", st); e = launch_slice10(Ht_hi, Ht_lo, h->expoT, h->Htdig, din, h->d_pad, group_size, st); ps.done(); count_launches(2); }
        if (e != cudaSuccess) { rc = cuda_fail(e); break; }
        { ProfScope ps("slices", st); e = launch_slices(h->Hs, h->expo, h->Hdig8, h->Hdig10, din, h->d_pad, group_size, st); ps.done(); count_launches(2); }
        if (e != cudaSuccess) { rc = cuda_fail(e); break; }
        int sb = 0;
        if ((e = read_status(h, st, &sb)) != cudaSuccess) { rc = cuda_fail(e); break; }
        rc = status_from_bits(sb);
    } while (0);
    if (Hdev || Ht_hi || Ht_lo) {
        cudaStreamSynchronize(st);
        cudaFree(Hdev);
        cudaFree(Ht_hi);
        cudaFree(Ht_lo);
    }
    if (rc != JARQ_OK) {
        jarq_hessian_destroy(h);
        return rc;
    }
    *out = h;
    return JARQ_OK;
}

jarq_status jarq_objective(jarq_hessian *h, const float *W, const float *S, const uint8_t *Q,
                           const int32_t *Z, int dout, int bits, double *F_per_row,
                           void *stream) {
    if (!layer_args_ok(h, W, S, Q, Z, dout, bits) || (dout > 0 && !F_per_row))
        return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    DeviceGuard dg(h->device);
    if (!dg.ok()) return JARQ_ERR_CUDA;
    cudaStream_t st = (cudaStream_t)stream;
    LayerArgs la;
    jarq_status rc = layer_front(h, W, S, Q, Z, dout, bits, la, st);
    if (rc != JARQ_OK) return rc;
    Workspace &w = h->ws;
    CK(cudaMemsetAsync(h->dstatus, 0, sizeof(int), st));
    RUN("hr_full", 1, launch_tc_hr_full(w.mapR, h->mapH128, w.Hr, h->din, dout, w.p_pad, h->din, h->d_pad, h->dstatus, st));
    RUN("grad", 1, launch_grad(la.Q, la.Z, w.r, w.Hr, nullptr, w.L_final, dout, h->din, h->g, st));
    CK(cudaMemcpyAsync(F_per_row, w.L_final, (size_t)dout * sizeof(double), cudaMemcpyDefault, st));
    int sb = 0;
    CK(read_status(h, st, &sb));
    return status_from_bits(sb);
}

jarq_status jarq_residual_product(jarq_hessian *h, const float *W, const float *S,
                                  const uint8_t *Q, const int32_t *Z, int dout, int bits,
                                  float *HR, void *stream) {
    if (!layer_args_ok(h, W, S, Q, Z, dout, bits) || (dout > 0 && !HR)) return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    DeviceGuard dg(h->device);
    if (!dg.ok()) return JARQ_ERR_CUDA;
    cudaStream_t st = (cudaStream_t)stream;
    LayerArgs la;
    jarq_status rc = layer_front(h, W, S, Q, Z, dout, bits, la, st);
    if (rc != JARQ_OK) return rc;
    Workspace &w = h->ws;
    CK(cudaMemsetAsync(h->dstatus, 0, sizeof(int), st));
    RUN("hr_full", 1, launch_tc_hr_full(w.mapR, h->mapH128, w.Hr, h->din, dout, w.p_pad, h->din, h->d_pad, h->dstatus, st));
    CK(cudaMemcpyAsync(HR, w.Hr, (size_t)dout * h->din * sizeof(float), cudaMemcpyDefault, st));
    int sb = 0;
    CK(read_status(h, st, &sb));
    return status_from_bits(sb);
}

jarq_status jarq_refine_layer(jarq_hessian *h, const float *W, float *S, uint8_t *Q,
                              const int32_t *Z, int dout, int bits, const jarq_options *opt,
                              jarq_stats *stats, void *stream) {
    return refine_impl(h, W, S, Q, Z, dout, bits, opt, stats, stream, nullptr);
}

jarq_status jarq_fit_scales(jarq_hessian *h, const float *W, float *S, const uint8_t *Q,
                            const int32_t *Z, int dout, int bits, jarq_fit method, int passes,
                            double *F_before, double *F_after, void *stream) {
    if (!layer_args_ok(h, W, S, Q, Z, dout, bits)) return JARQ_ERR_ARG;
    if (method != JARQ_FIT_JOINT && method != JARQ_FIT_INDEPENDENT &&
        method != JARQ_FIT_COORDINATE)
        return JARQ_ERR_ARG;
    if (method == JARQ_FIT_COORDINATE && passes < 1) return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    DeviceGuard dg(h->device);
    if (!dg.ok()) return JARQ_ERR_CUDA;
    cudaStream_t st = (cudaStream_t)stream;
    LayerArgs la;
    jarq_status rc = layer_front(h, W, S, Q, Z, dout, bits, la, st, true);
    if (rc != JARQ_OK) return rc;
    Workspace &w = h->ws;
    const int p = dout, d = h->din, g = h->g, G = h->G;
    RUN("init_rows", 1, launch_init_rows(w.active, w.iters, w.accepted, w.ridge, w.rstat, p, st));
    RUN("slice_rows", 1, launch_slice_rows(la.W, w.wdig, w.wexp, p, d, h->d_pad, w.p_pad, g, st));
    RUN("proj", 1, launch_tc_proj(w.mapWd, h->mapD8, w.Phi, w.Plo, w.wexp, h->expo, p, w.p_pad, d,
                                  h->d_pad, g, h->dstatus, st));
    RUN("whw", 1, launch_whw(la.W, w.Phi, w.Plo, w.wHw, p, d, st));
    RUN("gram", 1, launch_tc_gram(w.mapC, h->mapD10, la.Q, la.Z, h->expo, nullptr, w.gram, p,
                                  w.p_pad, d, h->d_pad, g, bits, h->dstatus, st));
    RUN("rhs", 1, launch_rhs(la.Q, la.Z, w.Phi, w.Plo, nullptr, w.rhs, p, d, g, st));
    if (method == JARQ_FIT_JOINT) {
        jarq_options o = jarq_default_options();
        o.early_stop = 0;
        RUN("scale_solve", 1, launch_scale_solve(w.gram, w.rhs, w.wHw, la.S, w.L_prev, w.L_host,
                                                 w.active, w.iters, w.ridge, w.rstat, h->dstatus,
                                                 p, d, g, 1, false, o, st));
        CK(cudaMemcpyAsync(w.L_final, w.L_prev, p * sizeof(double), cudaMemcpyDeviceToDevice, st));
    } else {
        if (method == JARQ_FIT_INDEPENDENT)
            RUN("own_rhs", 1, launch_own_rhs(h->Hs, la.W, la.Q, la.Z, w.own, p, d, g, st));
        RUN("scale_fit", 1, launch_scale_fit(w.gram, w.rhs, w.own, w.wHw, la.S, w.L_host,
                                             w.L_final, p, G, (int)method, passes, st));
    }
    if (la.hS) CK(cudaMemcpyAsync(S, la.S, (size_t)p * G * sizeof(float), cudaMemcpyDeviceToHost, st));
    if (F_before) CK(cudaMemcpyAsync(F_before, w.L_host, p * sizeof(double), cudaMemcpyDefault, st));
    if (F_after) CK(cudaMemcpyAsync(F_after, w.L_final, p * sizeof(double), cudaMemcpyDefault, st));
    int sb = 0;
    CK(read_status(h, st, &sb));
    return status_from_bits(sb);
}

jarq_status jarq_multicode_probe(jarq_hessian *h, const float *W, const float *S,
                                 const uint8_t *Q, const int32_t *Z, int dout, int bits,
                                 int group, uint8_t *Q_search, int32_t *moves, int32_t *accepted,
                                 int32_t *changed, double *dF, void *stream) {
    if (!layer_args_ok(h, W, S, Q, Z, dout, bits) || group < 0 || group >= h->G) return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    DeviceGuard dg(h->device);
    if (!dg.ok()) return JARQ_ERR_CUDA;
    cudaStream_t st = (cudaStream_t)stream;
    LayerArgs la;
    jarq_status rc = layer_front(h, W, S, Q, Z, dout, bits, la, st, true);
    if (rc != JARQ_OK) return rc;
    Workspace &w = h->ws;
    const int p = dout, d = h->din, g = h->g, G = h->G;
    const int nsplit = target_splits(w.p_pad, g, G);
    RUN("slice_rows", 1, launch_slice_rows(la.W, w.wdig, w.wexp, p, d, h->d_pad, w.p_pad, g, st));
    RUN("proj", 1, launch_tc_proj(w.mapWd, h->mapD8, w.Phi, w.Plo, w.wexp, h->expo, p, w.p_pad, d,
                                  h->d_pad, g, h->dstatus, st));
    // T = sum_h s_h H_ih c_h: the phase product with H's own digits
    RUN("target", 1, launch_tc_target(w.mapC, h->mapD10, w.t_hi, w.t_lo, la.S, h->expo, nullptr, p,
                                      w.p_pad, h->d_pad, g, G, group, nsplit, 0, p, (1 << bits) - 1,
                                      h->dstatus, st));
    uint8_t *qo = reinterpret_cast<uint8_t *>(w.Hr);
    RUN("probe", 1, launch_probe(w.Phi, w.Plo, w.t_hi, w.t_lo, h->Hs, h->L64, la.S, la.Q, la.Z, qo,
                                 w.iters, w.accepted, w.ridge, w.L_final, p, w.p_pad, d, g, group,
                                 nsplit, (1 << bits) - 1, FLT_EPSILON, st));
    if (Q_search) CK(cudaMemcpyAsync(Q_search, qo, (size_t)p * g, cudaMemcpyDefault, st));
    if (moves) CK(cudaMemcpyAsync(moves, w.iters, p * sizeof(int32_t), cudaMemcpyDefault, st));
    if (accepted) CK(cudaMemcpyAsync(accepted, w.accepted, p * sizeof(int32_t), cudaMemcpyDefault, st));
    if (changed) CK(cudaMemcpyAsync(changed, w.ridge, p * sizeof(int32_t), cudaMemcpyDefault, st));
    if (dF) CK(cudaMemcpyAsync(dF, w.L_final, p * sizeof(double), cudaMemcpyDefault, st));
    int sb = 0;
    CK(read_status(h, st, &sb));
    return status_from_bits(sb);
}

jarq_status jarq_refine_layer_mu(jarq_hessian *h, const float *W, float *S, uint8_t *Q,
                                 const int32_t *Z, int dout, int bits, const float *K,
                                 const float *XX, float mu, float nu2, const jarq_options *opt,
                                 jarq_stats *stats, void *stream) {
    if (!(mu >= 0.f && mu <= 1.f) || !(nu2 >= 0.f) || !isfinite(nu2)) return JARQ_ERR_ARG;
    if (mu == 1.f) return refine_impl(h, W, S, Q, Z, dout, bits, opt, stats, stream, nullptr);
    if (!K || !XX) return JARQ_ERR_ARG;
    MuTarget t{K, XX, mu, nu2};
    return refine_impl(h, W, S, Q, Z, dout, bits, opt, stats, stream, &t);
}

}  // extern "C"

namespace {

jarq_status refine_impl(jarq_hessian *h, const float *W, float *S, uint8_t *Q, const int32_t *Z,
                        int dout, int bits, const jarq_options *opt, jarq_stats *stats,
                        void *stream, const MuTarget *mt) {
    if (!layer_args_ok(h, W, S, Q, Z, dout, bits)) return JARQ_ERR_ARG;
    jarq_options o = opt ? *opt : jarq_default_options();
    if (o.max_iters < 0 || !(o.ridge >= 0.f) || !(o.rcond >= 0.f) || !(o.eps >= 0.f))
        return JARQ_ERR_ARG;
    if (dout == 0) return JARQ_OK;
    DeviceGuard dg(h->device);
    if (!dg.ok()) return JARQ_ERR_CUDA;
    cudaStream_t st = (cudaStream_t)stream;
    LayerArgs la;
    jarq_status rc = layer_front(h, W, S, Q, Z, dout, bits, la, st, true);
    if (rc != JARQ_OK) return rc;
    Workspace &w = h->ws;
    const int p = dout, d = h->din, g = h->g, G = h->G, qmax = (1 << bits) - 1;
    RUN("init_rows", 1, launch_init_rows(w.active, w.iters, w.accepted, w.ridge, w.rstat, p, st));
    const ResidualView rv = rview(h);
    const int nsplit = target_splits(w.p_pad, g, G);
    // chains of the sweep: the row tiles split into nchain contiguous ranges
    // only when one phase product needs more than one wave of CTAs (the
    // chains then fill each other's last wave); otherwise a single chain
    // with programmatic launches is faster.  Two chains: on the 14336-row
    // layer three were 2 % faster and four slower.
    const int tiles = (p + 127) / 128;
    const int waves = (tiles * (g / 64) * nsplit + num_sms() - 1) / num_sms();
    int nchain = (tiles >= kSweepSplitTiles && waves > 1) ? 2 : 1;
    if (nchain > kMaxChains) nchain = kMaxChains;
    if (nchain > tiles) nchain = tiles;
    if (nchain < 1) nchain = 1;
    int chain_row[kMaxChains + 1];
    for (int c = 0; c <= nchain; ++c) chain_row[c] = c == nchain ? p : (tiles * c / nchain) * 128;
    for (int c = 0; c < nchain - 1; ++c) {
        if (!h->aux[c]) {
            CK(cudaStreamCreateWithFlags(&h->aux[c], cudaStreamNonBlocking));
            CK(cudaEventCreateWithFlags(&h->ev_join[c], cudaEventDisableTiming));
        }
        if (!h->ev_fork) CK(cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming));
    }
    // target projection P = W H, w^T H w and the folded Pt, once per call
    RUN("slice_rows", 1, launch_slice_rows(la.W, w.wdig, w.wexp, p, d, h->d_pad, w.p_pad, g, st));
    RUN("proj", 1, launch_tc_proj(w.mapWd, h->mapD8, w.Phi, w.Plo, w.wexp, h->expo, p, w.p_pad, d,
                                  h->d_pad, g, h->dstatus, st));
    RUN("whw", 1, launch_whw(la.W, w.Phi, w.Plo, w.wHw, p, d, st));
    if (mt) {
        // mu-target: P <- H w_corr and w^T H w <- ||y(mu)||^2 from the two
        // extra projections W XX and W K^T (Pt's buffers hold them until
        // the folded projection is formed)
        rc = mu_projection(h, la.W, p, *mt, st);
        if (rc != JARQ_OK) return rc;
    }
    RUN("ptilde", 2, launch_ptilde(w.mapPd, h->mapRi, w.Phi, w.Plo, w.wdig, w.wexp, h->rexp, w.Pt_hi,
                                   w.Pt_lo, p, w.p_pad, d, h->d_pad, g, h->dstatus, st));
    for (int k = 1; k <= o.max_iters; ++k) {
        // with the early stop off every row is refined (a row marked numerical
        // is skipped by the solve and Babai), so the Gram and the right-hand
        // side need not read the active flags
        const int *act_es = o.early_stop ? w.active : nullptr;
        RUN("gram", 1, launch_tc_gram(w.mapC, h->mapD10, la.Q, la.Z, h->expo, act_es, w.gram, p,
                                      w.p_pad, d, h->d_pad, g, bits, h->dstatus, st));
        RUN("rhs", 1, launch_rhs(la.Q, la.Z, w.Phi, w.Plo, act_es, w.rhs, p, d, g, st));
        double *L_out = (k == 1 && stats && stats->L_host) ? w.L_host : nullptr;
        RUN("scale_solve", 1, launch_scale_solve(w.gram, w.rhs, w.wHw, la.S, w.L_prev, L_out,
                                                 w.active, w.iters, w.ridge, w.rstat, h->dstatus,
                                                 p, d, g, k, false, o, st));
        // The phase product reads the active flags only with the early stop
        // on (to skip tiles whose rows all stopped); a row marked numerical
        // by the scale solve is skipped by Babai, and its partials go unread.
        // The sweep.  Rows are independent, so the row tiles may form several
        // ranges, each with its own chain of phase products and Babai steps
        // on its own stream: one chain's Babai step runs on the SMs that
        // another chain's phase product leaves free, and each chain's launch
        // gaps are filled by the others' work.  Programmatic launch only for
        // a single chain: an early-launched grid waits on its SMs, which the
        // other chains' kernels need.
        const bool pdl = nchain == 1;
        ChainJoin join{h, st, 0};
        if (nchain > 1) {
            CK(cudaEventRecord(h->ev_fork, st));
            for (int c = 0; c < nchain - 1; ++c) {
                CK(cudaStreamWaitEvent(h->aux[c], h->ev_fork, 0));
                join.n = c + 1;
            }
        }
        for (int i = 0; i < G; ++i) {
            for (int c = 0; c < nchain; ++c) {
                cudaStream_t sc = c == 0 ? st : h->aux[c - 1];
                const int r0 = chain_row[c], r1 = chain_row[c + 1];
                RUN_ON("target", 1, sc,
                       launch_tc_target(w.mapC, h->mapHt, w.t_hi, w.t_lo, la.S, h->expoT,
                                        o.early_stop ? w.active : nullptr, p, w.p_pad,
                                        h->d_pad, g, G, i, nsplit, r0, r1 - r0, qmax,
                                        h->dstatus, sc, pdl));
                RUN_ON("babai", 1, sc,
                       launch_babai(w.t_hi, w.t_lo, w.Pt_hi, w.Pt_lo, nsplit, h->Lf, la.S, la.Q,
                                    la.Z, rv, w.active, w.accepted, h->dstatus, p, g, i, qmax,
                                    o.eps, r0, r1, sc, pdl));
            }
        }
        join.n = 0;
        for (int c = 0; c < nchain - 1; ++c) {
            CK(cudaEventRecord(h->ev_join[c], h->aux[c]));
            CK(cudaStreamWaitEvent(st, h->ev_join[c], 0));
        }
    }
    // objective of the returned state (and of the input state when K = 0)
    const bool want_final = stats && stats->L_final;
    const bool want_host0 = stats && stats->L_host && o.max_iters == 0;
    if (want_final || want_host0) {
        RUN("gram", 1, launch_tc_gram(w.mapC, h->mapD10, la.Q, la.Z, h->expo, nullptr, w.gram, p,
                                      w.p_pad, d, h->d_pad, g, bits, h->dstatus, st));
        RUN("rhs", 1, launch_rhs(la.Q, la.Z, w.Phi, w.Plo, nullptr, w.rhs, p, d, g, st));
        RUN("scale_solve", 1, launch_scale_solve(w.gram, w.rhs, w.wHw, la.S, w.L_prev, w.L_final,
                                                 w.active, w.iters, w.ridge, w.rstat, h->dstatus,
                                                 p, d, g, 0, true, o, st));
        if (want_host0)
            CK(cudaMemcpyAsync(w.L_host, w.L_final, p * sizeof(double), cudaMemcpyDeviceToDevice, st));
    }
    if (la.hS) CK(cudaMemcpyAsync(S, la.S, (size_t)p * G * sizeof(float), cudaMemcpyDeviceToHost, st));
    if (la.hQ) CK(cudaMemcpyAsync(Q, la.Q, (size_t)p * d, cudaMemcpyDefault, st));
    if (stats) {
        if (stats->L_host) CK(cudaMemcpyAsync(stats->L_host, w.L_host, p * sizeof(double), cudaMemcpyDefault, st));
        if (stats->L_final) CK(cudaMemcpyAsync(stats->L_final, w.L_final, p * sizeof(double), cudaMemcpyDefault, st));
        if (stats->iters) CK(cudaMemcpyAsync(stats->iters, w.iters, p * sizeof(int), cudaMemcpyDefault, st));
        if (stats->accepted) CK(cudaMemcpyAsync(stats->accepted, w.accepted, p * sizeof(int), cudaMemcpyDefault, st));
        if (stats->ridge_hits) CK(cudaMemcpyAsync(stats->ridge_hits, w.ridge, p * sizeof(int), cudaMemcpyDefault, st));
        if (stats->row_status) CK(cudaMemcpyAsync(stats->row_status, w.rstat, p * sizeof(int), cudaMemcpyDefault, st));
    }
    int sb = 0;
    CK(read_status(h, st, &sb));
    return status_from_bits(sb);
}

}  // namespace
