/*
 * jarq.h -- C ABI of the GB300 (sm_103a) JARQ layer-refinement library.
 *
 * JARQ (Joint Alternating Refinement for Quantization) refines a group-wise
 * uniformly quantized linear layer.  Given the layer's weights W, the
 * calibration Hessian H = A^T A (A = [X; nu I], Sec. 3.2, Eq. strict_target)
 * and a host quantizer's scales S, integer codes Q and zero points Z
 * (Sec. 3.1, Eq. quantized_group), it minimises the per-row objective
 *
 *     F_j = (w_j - what_j)^T H (w_j - what_j),  what_j = D_{s_j}(q_j - z_j)
 *
 * (Eq. bbmils_columns with the main target Y = A W) by alternating
 *   (a) a joint least-squares fit of all G scales of a row, solved by
 *       Cholesky on the G x G normal equations (Sec. 3.3.1, Eqs.
 *       scale_design / scale_normal_equations, with the ridge safeguard of
 *       App. E "Solving for scales"), and
 *   (b) one Gauss-Seidel sweep of bounded Babai nearest-plane proposals over
 *       the groups, each kept only if it strictly lowers the objective
 *       (Sec. 3.3.2, Eqs. conditional_residual, group_qr, babai_update).
 * Bit width, groups and zero points never change.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Layout: W is float32 [dout][din] row-major (row j is the paper's column
 *   w_j); S is float32 [dout][G]; Q is uint8 [dout][din]; Z is int32
 *   [dout][G]; H is float32 [din][din]; G = din / group_size.
 * - Pointers may be device memory or host memory (pageable or pinned).
 *   Host buffers are staged through library-owned device buffers; device
 *   buffers are used in place, except a device Q that is not 16-byte
 *   aligned, which is staged like host memory.  The caller owns every
 *   buffer it passes.
 * - `stream` is a cudaStream_t passed as void* (NULL = the legacy default
 *   stream).  Work is enqueued on it in order.  Calls return after the work
 *   they enqueued has finished and its status has been read back.
 * - Errors are reported as jarq_status values; no exception or abort crosses
 *   the ABI.  On JARQ_ERR_ARG nothing is enqueued and no buffer is touched.
 * - A handle is not thread-safe: do not use one handle from two host threads
 *   or on two streams at the same time.  Different handles are independent.
 */
#ifndef JARQ_H_
#define JARQ_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum jarq_status {
    JARQ_OK = 0,
    JARQ_ERR_ARG = 1,        /* invalid argument (size, pointer, range)        */
    JARQ_ERR_NOT_SPD = 2,    /* a diagonal block H_ii is not positive definite */
    JARQ_ERR_NUMERICAL = 3,  /* a scale system failed even with the ridge      */
    JARQ_ERR_CUDA = 4,       /* a CUDA runtime or driver call failed           */
    JARQ_ERR_TIMEOUT = 5,    /* a bounded device wait gave up; outputs invalid  */
    JARQ_ERR_NOMEM = 6       /* device allocation failed                       */
} jarq_status;

/* Opaque prepared Hessian: symmetrised H, its split-precision copy for the
 * tensor cores and the per-group Cholesky factors R_i (H_ii = R_i^T R_i) with
 * their inverses.  Sec. 3.3.2 (Eq. group_qr) precomputes these once and
 * reuses them for every output row and iteration; R_i equals the paper's
 * thin-QR factor up to row signs, to which Babai is invariant.  Library-owned;
 * also caches the refinement workspaces, sized by the largest dout seen. */
typedef struct jarq_hessian jarq_hessian;

/* Solver settings (App. E "Numerical Updates and Stopping").  Fill with
 * jarq_default_options() and override fields. */
typedef struct jarq_options {
    int   max_iters;     /* K, the iteration budget (paper: 3).  0 returns the host state. */
    int   early_stop;    /* 1: per-row stop of Eq. strict_stopping for k >= 2; 0: run K iterations */
    float tau_rel;       /* relative stop threshold tau (1e-5)                    */
    float tau_abs;       /* absolute stop threshold tau (1e-5)                    */
    float ridge;         /* lambda added when the Gram matrix is nearly singular (1e-4) */
    float rcond;         /* r_cond of the near-singularity test (1e-10)           */
    float eps;           /* eps_fp: FP32 machine epsilon; small-scale skip threshold */
    int   ridge_accept;  /* 1: keep a ridge-stabilised solve only if it does not raise F_j,
                            else keep the previous scales (App. G Remark ridge-acceptance);
                            0 (default): keep every solve, as the paper's runs do */
    int   fixed_grid;    /* 1: keep the host scales, update only the codes -- the "Fixed"
                            arm of App. "Fixed-Grid versus Joint Refinement"; each iteration
                            still evaluates L^(k) for the early stop.  0 (default): JARQ */
} jarq_options;

/* Scale fits of jarq_fit_scales (App. "Joint Scale Fitting"). */
typedef enum jarq_fit {
    JARQ_FIT_JOINT = 0,        /* the joint normal equations (Eq. scale_normal_equations) */
    JARQ_FIT_INDEPENDENT = 1,  /* each group on its own contribution (Eq. independent-fit) */
    JARQ_FIT_COORDINATE = 2    /* cyclic exact coordinate descent on the scales */
} jarq_fit;

/* Element types of jarq_dequantize's output. */
typedef enum jarq_dtype { JARQ_F32 = 0, JARQ_F16 = 1, JARQ_BF16 = 2 } jarq_dtype;

/* Per-row statistics.  Every pointer may be NULL (not collected) and may be
 * host or device memory; arrays have dout entries.
 *   L_host     : objective F_j of the input state (S, Q)            [double]
 *   L_final    : objective F_j of the returned state                 [double]
 *   iters      : scale updates performed (<= max_iters)              [int32]
 *   accepted   : Babai proposals accepted                            [int32]
 *   ridge_hits : scale solves that needed the ridge                  [int32]
 *   row_status : JARQ_OK or JARQ_ERR_NUMERICAL for that row          [int32]  */
typedef struct jarq_stats {
    double  *L_host;
    double  *L_final;
    int32_t *iters;
    int32_t *accepted;
    int32_t *ridge_hits;
    int32_t *row_status;
} jarq_stats;

/* Default options: K = 3, early stop on, tau = 1e-5, ridge 1e-4,
 * rcond 1e-10, eps = FLT_EPSILON (App. E), ridge acceptance off. */
jarq_options jarq_default_options(void);

/* Prepare a Hessian for refinement (Sec. 3.3.2, Eq. group_qr; App. G.7
 * "Shared preprocessing").
 *   H          : float32 [din][din], host or device; symmetrised as (H+H^T)/2.
 *   din        : input width, > 0, multiple of group_size, at most
 *                128 groups.
 *   group_size : g, 64 or 128 (the paper's group sizes that fit the
 *                tensor-core tiles and the Babai kernel's shared memory).
 *   nu2        : added to the diagonal (the paper's nu^2, Eq. strict_target);
 *                pass 0 when H already contains its damping.
 *   out        : receives the new handle (unchanged on error).
 * Returns JARQ_ERR_NOT_SPD if some H_ii is not positive definite,
 * JARQ_ERR_ARG for bad sizes or a NULL pointer. */
jarq_status jarq_prepare_hessian(const float *H, int din, int group_size, float nu2,
                                 jarq_hessian **out, void *stream);

/* Refine one layer in place: K iterations of joint scale fit + Babai sweep
 * (Sec. 3.3; App. E "Order of updates", "Early stopping", "Small scales").
 * Each solved scale is stored as float32, the precision of the paper's scale
 * solve (App. E "Solving for scales"), before the codes are updated.
 *   h      : prepared Hessian for this layer's input (din, group size).
 *   W      : float32 [dout][din], original weights (read only).
 *   S      : float32 [dout][G], host scales in, refined signed scales out.
 *   Q      : uint8 [dout][din], codes in [0, 2^bits - 1]; refined in place.
 *   Z      : int32 [dout][G], zero points in [0, 2^bits - 1]; read only.
 *   dout   : output rows, >= 0 (0 is a no-op).
 *   bits   : b, 1 <= b <= 8.
 *   opt    : solver settings (NULL = jarq_default_options()).
 *   stats  : optional per-row statistics (NULL = none).
 * Rows are independent; a row whose scale system fails even with the ridge
 * keeps its last state and is marked JARQ_ERR_NUMERICAL in row_status, the
 * other rows finish, and the call returns JARQ_ERR_NUMERICAL.  Codes or zero
 * points outside [0, 2^bits - 1] return JARQ_ERR_ARG before any update. */
jarq_status jarq_refine_layer(jarq_hessian *h, const float *W, float *S, uint8_t *Q,
                              const int32_t *Z, int dout, int bits,
                              const jarq_options *opt, jarq_stats *stats, void *stream);

/* Refinement on the propagation-corrected target (App. "Propagation-
 * Corrected Targets and QEP", Eq. mu-target): the activation part of the
 * target becomes Y*(mu) = (1 - mu) X W + mu X~ W, with X the layer's
 * full-precision inputs and X~ the inputs after the quantized preceding
 * layers; mu = 1 is the main target (this call is then jarq_refine_layer and
 * K, XX are not read).  Equivalently (Eq. w-corr) the main problem on
 * W_corr = W + (1 - mu) H^{-1} X~^T (X - X~) W plus a per-row constant; the
 * library never forms H^{-1}: it replaces H w by H w_corr = mu H w +
 * (1 - mu)(K w + nu2 w) and w^T H w by ||y(mu)||^2, both from exact
 * tensor-core projections, and runs the same loop.  S, Q and the reported
 * objectives (stats L_host, L_final) are those of the mu-target, constant
 * included; early stopping uses them.
 *   h, W, S, Q, Z, dout, bits, opt, stats, stream : as jarq_refine_layer; h
 *        must be prepared from H = X~^T X~ + nu2 I.
 *   K    : float32 [din][din], host or device: X~^T X, normalised like H.
 *   XX   : float32 [din][din], host or device: X^T X, normalised like H.
 *   mu   : in [0, 1].
 *   nu2  : the nu^2 contained in the prepared H, >= 0 and finite.
 * The first call with mu < 1 allocates the handle's digit planes for K and
 * XX (6 din^2 bf16, kept until the handle is destroyed).  Errors as
 * jarq_refine_layer; mu outside [0, 1], a non-finite or negative nu2, or a
 * NULL K or XX with mu < 1 return JARQ_ERR_ARG. */
jarq_status jarq_refine_layer_mu(jarq_hessian *h, const float *W, float *S, uint8_t *Q,
                                 const int32_t *Z, int dout, int bits, const float *K,
                                 const float *XX, float mu, float nu2, const jarq_options *opt,
                                 jarq_stats *stats, void *stream);

/* Per-row objective F_j = r_j^T H r_j, r_j = w_j - D_{s_j}(q_j - z_j)
 * (Sec. 3.2, Eq. bbmils_columns), written as double to F_per_row[dout]
 * (host or device).  Same layouts and checks as jarq_refine_layer. */
jarq_status jarq_objective(jarq_hessian *h, const float *W, const float *S, const uint8_t *Q,
                           const int32_t *Z, int dout, int bits, double *F_per_row,
                           void *stream);

/* The residual product H r_j of every row, r_j = w_j - D_{s_j}(q_j - z_j),
 * written as float32 to HR[dout][din] (host or device): the group slices
 * (H r_j)_i of Sec. 3.3.2, Eq. conditional_residual, for every group at
 * once.  It is computed by the split-precision tensor-core kernel behind
 * jarq_objective (the refinement's sweep forms its Babai targets with the
 * exact folded phase product instead), and it exists so that tests can
 * compare that contraction element by element with a reference.  Same
 * layouts and checks as jarq_refine_layer. */
jarq_status jarq_residual_product(jarq_hessian *h, const float *W, const float *S,
                                  const uint8_t *Q, const int32_t *Z, int dout, int bits,
                                  float *HR, void *stream);

/* ---- mechanism ablations (App. "Refinement Mechanisms", Tab. mechanism-summary (a)) ----
 * Same layouts, staging and code checks as jarq_refine_layer. */

/* Fit all scales of every row for the given codes with one of the three fits
 * that the paper compares (App. "Joint Scale Fitting"):
 *   JARQ_FIT_JOINT        the joint least-squares fit (Sec. 3.3.1), with the
 *                         ridge safeguard of App. E;
 *   JARQ_FIT_INDEPENDENT  s_i = c_i^T H_ii w_i / c_i^T H_ii c_i, each group on
 *                         its own contribution (Eq. independent-fit);
 *   JARQ_FIT_COORDINATE   `passes` cyclic passes over the groups, each scale
 *                         moved to the exact minimiser of F along it, starting
 *                         from the input S.
 * A group whose codes all equal its zero point keeps its scale in the last
 * two.  S is overwritten with the fitted float32 scales; F_before / F_after
 * (optional, [dout] double, host or device) receive the objective of the
 * input and of the fitted scales.  passes >= 1 for JARQ_FIT_COORDINATE. */
jarq_status jarq_fit_scales(jarq_hessian *h, const float *W, float *S, const uint8_t *Q,
                            const int32_t *Z, int dout, int bits, jarq_fit method, int passes,
                            double *F_before, double *F_after, void *stream);

/* Multi-code probe of one group (App. "Multi-Code Updates"): for every row,
 * with the scales and the other groups fixed, single-code updates of group
 * `group` (each coordinate in order moved to its best code when that
 * strictly lowers F; full passes until a pass moves nothing), then one
 * bounded Babai proposal from that single-code-stationary state (Eq.
 * babai_update), accepted iff it strictly lowers F.  Decisions are taken in
 * float64.  Nothing is written back to S or Q.  Outputs (optional, host or
 * device): Q_search [dout][g] uint8, the codes after the search; moves
 * [dout], the single-code moves made; accepted [dout], 1 if the Babai
 * proposal strictly lowers F; changed [dout], codes the proposal changes;
 * dF [dout] double, its change of F.  Rows with |s| <= FLT_EPSILON are
 * skipped (all outputs 0, codes unchanged). */
jarq_status jarq_multicode_probe(jarq_hessian *h, const float *W, const float *S,
                                 const uint8_t *Q, const int32_t *Z, int dout, int bits,
                                 int group, uint8_t *Q_search, int32_t *moves, int32_t *accepted,
                                 int32_t *changed, double *dF, void *stream);

/* ---- write-back of a refined layer (device memory only) ----
 * These post-passes act on a layer already in device memory; host pointers
 * return JARQ_ERR_ARG.  They allocate nothing and return after their work
 * has finished.  Codes and zero points must lie in [0, 2^bits - 1]
 * (JARQ_ERR_ARG otherwise, before any change). */

/* Negative-scale canonicalisation (App. E "Representing Negative Scales",
 * Eq. canonicalization): for every group with s < 0, s' = -s,
 * q' = qmax - q, z' = qmax - z, which leaves s (q - z) unchanged.
 *   S [dout][G] float32, Q [dout][din] uint8, Z [dout][G] int32: in place. */
jarq_status jarq_canonicalize(float *S, uint8_t *Q, int32_t *Z, int dout, int din,
                              int group_size, int bits, void *stream);

/* The returned weights what = s (q - z) (Sec. 3.1, Eq. quantized_group),
 * exact before one round-to-nearest-even to `dtype`, written to
 * W_out [dout][din] (App. E: the refined weights are cast to the model's
 * weight dtype). */
jarq_status jarq_dequantize(const float *S, const uint8_t *Q, const int32_t *Z, int dout, int din,
                            int group_size, int bits, jarq_dtype dtype, void *W_out, void *stream);

/* b-bit codes packed per row into a little-endian bit stream: code k of a
 * row occupies bits [k b, k b + b), cut into 32-bit words, the last word
 * zero-padded.  packed [dout][ceil(din * bits / 32)] uint32. */
jarq_status jarq_pack_codes(const uint8_t *Q, int dout, int din, int bits, uint32_t *packed,
                            void *stream);

/* ---- calibration Hessian (device memory only) ----
 * H <- H + scale * X^T X, the activation part of the Hessian H = A^T A of
 * the augmented design A = [X~; nu I] (Sec. 3.2, Eq. strict_target; the
 * paper writes H = X~^T X~ + nu^2 I out in its appendix on
 * propagation-corrected targets).  nu^2 I is added by jarq_prepare_hessian.
 * Called once per batch of calibration tokens, it accumulates H over an
 * activation stream.
 *   X     : device, float16 [n][d] row-major, one token per row (the layer's
 *           inputs as the preceding quantized layers produce them), 16-byte
 *           aligned; d a multiple of 8, 8 <= d <= 65536.  Not modified.
 *   n     : tokens in this batch, >= 0 (0: nothing to do, H untouched).
 *   scale : finite multiplier of the batch's product (1 for the paper's H).
 *   H     : device, float32 [d][d] row-major, 16-byte aligned, read and
 *           written in place;
 *           every element, both triangles, becomes
 *           fl(H[i][j] + scale * sum_t X[t][i] X[t][j]), so a symmetric H
 *           stays exactly symmetric.  Must not overlap X.
 * Precision: the fp16 products are exact (the paper forms its products from
 * FP16 activations in FP32, App. "Metrics"); they are summed in float32 on
 * the tensor cores over blocks of 512 tokens, the block sums in float32,
 * and the result is added to H with one rounding.
 * Errors: JARQ_ERR_ARG (sizes, a non-finite scale, null, host or misaligned
 * pointers; nothing enqueued), JARQ_ERR_TIMEOUT (a bounded device wait gave
 * up; H is then unspecified), JARQ_ERR_CUDA.  Returns after the update has
 * finished. */
jarq_status jarq_accumulate_hessian(const void *X, int n, int d, float scale, float *H,
                                    void *stream);

/* Per-row objective without any device allocation.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory when they need the objective -- serving processes that
 * reserve all device memory at start-up and forbid later allocations, and
 * callers that cannot afford the device-wide synchronisation an allocation
 * may cause.  It computes the same values as jarq_objective.
 *   All buffers must be device memory of the handle's GPU (host pointers and
 *   buffers on another GPU return JARQ_ERR_ARG; staging host memory would
 *   allocate).  The prepared handle h comes from jarq_prepare_hessian, which
 *   allocates once, up front.  The caller's current device is restored
 *   before the call returns.
 *   Limit: ceil(dout/128)*128 * ceil(din/128)*128 <= 2^20 (for example a
 *   1024 x 1024 layer); larger layers return JARQ_ERR_ARG.
 *   Scratch: one statically sized device array (about 16 MiB) that every GPU
 *   loading the library holds until the process exits.  All calls share it
 *   and it keeps the last call's contents; the call clears what must start at
 *   zero.  Calls that overlap on the GPU (from two streams or two host
 *   threads) race on it: serialise them.
 *   The first call on a device looks up the array's device address once.
 *   Synchronous: the call waits on `stream` after checking the codes and
 *   again at the end, and reads the status on the host; it returns after
 *   the results are in F_per_row. */
jarq_status jarq_objective_noalloc(jarq_hessian *h, const float *W, const float *S,
                                   const uint8_t *Q, const int32_t *Z, int dout, int bits,
                                   double *F_per_row, void *stream);

/* Input width and group size of a prepared handle (0 for NULL). */
int jarq_hessian_din(const jarq_hessian *h);
int jarq_hessian_group_size(const jarq_hessian *h);

/* Release a handle and its workspaces (NULL is a no-op).  Synchronises the
 * device first so no enqueued work still uses them. */
void jarq_hessian_destroy(jarq_hessian *h);

/* Static, human-readable name of a status. */
const char *jarq_status_string(jarq_status s);

/* ---- Instrumentation (no counterpart in the paper) -------------------------
 * Used by the benchmark to time individual kernels on the stream they run
 * on.  When enabled, the library records a CUDA event pair around every
 * kernel launch it makes; durations are accumulated per kernel name when the
 * enclosing call synchronises.  Names: "validate", "residual", "init_rows",
 * "hr_full", "grad", "gram", "scale_solve", "phase_hr", "babai",
 * "symmetrize", "group_factor", "slices", "slice_rows", "proj", "whw", "rhs",
 * "htilde", "ptilde", "target", "syrk", "mu_combine", "own_rhs", "scale_fit",
 * "probe".  Not thread-safe. */
void jarq_profile_enable(int on);
void jarq_profile_reset(void);
/* Accumulated launches and total device milliseconds of one kernel name since
 * the last reset; returns 0 on success, -1 for an unknown name. */
int jarq_profile_read(const char *kernel, long long *launches, double *total_ms);
/* Number of kernels this library has launched since it was loaded. */
long long jarq_launch_count(void);

/* Test hook for the bounded device waits (no counterpart in the paper).
 * Every wait of the library's kernels on a barrier gives up after a fixed
 * number of polls; the kernel then records the timeout, finishes its copies
 * in flight and returns, and the call reports JARQ_ERR_TIMEOUT.  This call
 * launches one thread that waits on a barrier nothing completes, with a
 * short poll limit, and returns the status the same path produces:
 * JARQ_ERR_TIMEOUT when it works.  The CUDA context stays usable.  `stream`
 * as for every entry point; returns after the stream work has finished. */
jarq_status jarq_selftest_wait_timeout(void *stream);

#ifdef __cplusplus
}
#endif

#endif /* JARQ_H_ */
