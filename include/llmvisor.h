/*
 * llmvisor.h -- C ABI of the GB300 (sm_103a) implementation of LLMVisor's
 * batched latency attribution.
 *
 * The model (Section 2, "Problem formulation", and Section 2.1, Eq. 1):
 * a batch B of requests has latency
 *     T_B = beta + a1*sum_i p_i + a2*sum_i c_i + a3*sum_i p_i^2 + a4*sum_i |B|
 * with four coefficient sets, one per (phase, regime): prefill or decode, and
 * memory-bound or compute-bound.  p_i is the number of tokens request i
 * processes this step, c_i the number of context tokens whose KV entries it
 * loads.  T_B splits into additive, per-request shares t_i with
 * sum_i t_i = T_B, and shares roll up per tenant: L_u = sum_{i: u(i)=u} t_i.
 *
 * Readings of the paper used throughout (it leaves these open):
 *  - sum_i |B| is taken literally: it equals n^2 for a batch of n requests.
 *  - A batch is a prefill batch if any request in it is a prefill.
 *  - Regime: compute-bound iff S1 = sum_i p_i >= split[phase] (tie -> compute).
 *  - Share: t_i = beta/n + a1 p_i + a2 c_i + a3 p_i^2 + a4 n (the fixed cost and
 *    the n^2 term are split equally; slope terms follow their request).
 *  - Empty batch: T = 0, segment (decode, memory), no shares.
 *  - Units: seconds, coefficients in seconds per raw feature unit.
 *
 * Conventions for every call:
 *  - Every array argument is DEVICE memory owned by the caller, unless stated.
 *    Structs (lv_arch, lv_model, lv_batches, lv_fit_report) live in HOST memory
 *    and are copied at the call; device pointers inside lv_batches are the
 *    caller's.  Opaque handles (lv_ctx, lv_tenant_acc) are owned by the library.
 *  - stream is a cudaStream_t (NULL = legacy default stream).  Calls are
 *    asynchronous with respect to the host unless stated.
 *  - Argument errors are detected on the host and returned before anything is
 *    launched (LV_EINVAL, LV_EOVERFLOW).  Data errors found on the device
 *    (non-monotone offsets, negative p or c, phase not 0/1, tenant out of range,
 *    offsets[n_batch] != n_req) never cause an out-of-bounds access: kernels
 *    clamp and record LV_EDATA in the context's sticky status word, which
 *    lv_ctx_status() reports.  CUDA failures return LV_ECUDA.
 *  - Alignment: request arrays (p, c, phase, tenant) and offsets must be
 *    16-byte aligned (so that kernels may read them with 16-byte vector loads),
 *    fp64 outputs 8-byte aligned; otherwise LV_EINVAL.
 *  - One lv_ctx must not be used from two host threads at once.
 *  - CUDA graphs: lv_features, lv_batch_latency, lv_attribute,
 *    lv_attribute_step, lv_tenant_acc_reset, lv_tenant_accumulate,
 *    lv_tenant_totals, lv_whatif
 *    and lv_whatif_admit may be captured into a CUDA graph once an uncaptured call with
 *    the same context, model and sizes has run (it creates the context's
 *    buffers and caches the kernel configuration; a capture never allocates).
 *    The context's ordering events are then recorded and waited for by the
 *    graph itself at each replay; library timing (lv_ctx_set_timing) skips
 *    captured launches.  lv_fit, lv_ctx_status and lv_tenant_acc_export /
 *    import synchronise and cannot be captured.
 */
#ifndef LLMVISOR_H
#define LLMVISOR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t lv_status;
#define LV_OK 0
#define LV_EINVAL (-1)     /* bad argument (null/unaligned pointer, bad size, bad arch) */
#define LV_EOVERFLOW (-2)  /* an int64 feature or constant would overflow */
#define LV_ENODATA (-3)    /* fit group with fewer batches than coefficients */
#define LV_ESINGULAR (-4)  /* fit group whose normal equations are singular */
#define LV_ECUDA (-5)      /* a CUDA runtime call failed */
#define LV_EDATA (-6)      /* invalid input data seen on the device (sticky) */
#define LV_ENOMEM (-7)     /* device allocation failed */
#define LV_ETIMEOUT (-8)   /* a bounded wait inside a kernel ran out (lv_accuracy, or lv_ctx_status after a serving-step launch) */

/* Model architecture; integers only.  tp is the modelled tensor-parallel degree
 * (an arithmetic input: constants are per rank).  kv_bytes is the KV-cache
 * element size.  tp must divide n_q_heads, n_kv_heads and ffn_dim. */
typedef struct {
    int32_t n_layers, d_model, n_q_heads, n_kv_heads, head_dim, ffn_dim;
    int32_t weight_bytes, kv_bytes, tp;
} lv_arch;

/* One coefficient set of Eq. 1, in seconds per raw unit. */
typedef struct {
    double beta, a1, a2, a3, a4;
} lv_coef;

/* The piecewise model: seg[phase][regime], phase 0 = decode, 1 = prefill;
 * regime 0 = memory-bound, 1 = compute-bound (Section 2.1: two segments per
 * phase, four coefficient sets in all).  split[phase] is the threshold on
 * S1 = sum_i p_i at which the regime becomes compute-bound. */
typedef struct {
    lv_coef seg[2][2];
    int64_t split[2];
} lv_model;

/* A set of batches in CSR form.  All pointers are DEVICE pointers.
 *  p[n_req], c[n_req], phase[n_req] (0 decode / 1 prefill), tenant[n_req]
 *  (0..n_tenants-1; may be NULL where no tenant roll-up is asked for),
 *  offsets[n_batch+1] with offsets[0] = 0, non-decreasing, offsets[n_batch] = n_req.
 *  Batch b holds requests offsets[b] .. offsets[b+1]-1. */
typedef struct {
    const int32_t *p, *c, *phase, *tenant;
    const int64_t *offsets;
    int64_t n_req, n_batch;
    int32_t n_tenants;
    int32_t reserved;
} lv_batches;

/* Per-group outcome of lv_fit, group g = phase*2 + regime. */
typedef struct {
    int64_t n[4];        /* batches in the group (empty batches excluded) */
    int32_t status[4];   /* LV_OK, LV_ENODATA or LV_ESINGULAR */
    int32_t dropped[4];  /* bit k set: coefficient k (0 beta .. 4 a4) not identifiable, reported as 0 */
    double ssr[4];       /* residual sum of squares of the returned coefficients */
    double r2[4];        /* 1 - ssr/sst */
} lv_fit_report;

/* Accuracy of predicted batch latencies (lv_accuracy). */
typedef struct {
    int64_t n;           /* batches with y > 0 (the samples) */
    double r2_ssr;       /* 1 - sum (y - T)^2 / sum (y - mean y)^2 */
    double r2_corr;      /* squared Pearson correlation of y and T */
    double mean_rel;     /* mean of |T - y| / y */
    double p50, p90, p99;  /* nearest-rank percentiles of |T - y| / y */
} lv_accuracy_report;

typedef struct lv_ctx lv_ctx;
typedef struct lv_tenant_acc lv_tenant_acc;

/* Arithmetic used for T and shares.  AUTO picks the exact fixed-point path
 * whenever every segment's coefficients fit it (see lv_attribute) and FP64
 * otherwise; FP64 forces double-precision evaluation. */
#define LV_ARITH_AUTO 0
#define LV_ARITH_FP64 1

/* Create a context on the current CUDA device.  It owns a small device scratch
 * area and a sticky status word.  Returns LV_ECUDA/LV_ENOMEM on failure. */
lv_status lv_ctx_create(lv_ctx **out);
void lv_ctx_destroy(lv_ctx *ctx);
/* Select LV_ARITH_AUTO (default) or LV_ARITH_FP64. */
lv_status lv_ctx_set_arith(lv_ctx *ctx, int32_t mode);
/* Synchronise `stream`, then return and clear the sticky device status
 * (LV_OK; LV_EDATA when a kernel met invalid input data since the last query;
 * LV_ETIMEOUT when a bounded wait inside the serving-step kernel of
 * lv_attribute / lv_attribute_step ran out, which takes precedence). */
lv_status lv_ctx_status(lv_ctx *ctx, void *stream);
/* Static description of a status code. */
const char *lv_status_string(lv_status s);
/* Measurement support (no counterpart in the paper).  `mask` selects which
 * request-streaming kernels the library brackets with CUDA events on the
 * launching stream: LV_TIME_TILES the tile kernel of lv_attribute /
 * lv_features / lv_fit / lv_whatif's candidate pass, LV_TIME_PAIRS the pair
 * kernel of lv_whatif; 0 (the default) none.  Other bits: LV_EINVAL.
 * lv_ctx_kernel_time synchronises those events, returns the summed
 * milliseconds and the number of launches since the previous query, and
 * resets the tally. */
#define LV_TIME_TILES 1
#define LV_TIME_PAIRS 2
lv_status lv_ctx_set_timing(lv_ctx *ctx, int32_t mask);
lv_status lv_ctx_kernel_time(lv_ctx *ctx, double *ms, int64_t *launches);
/* Failure-detection support (no counterpart in the paper): runs the grid-wide
 * barrier that lv_accuracy's kernel uses in a cooperative launch of two blocks,
 * one of which leaves without arriving, so that the other's bounded wait runs
 * out.  Returns LV_ETIMEOUT after a few seconds when the bound works as
 * designed (LV_OK would mean the barrier let a block through alone), with the
 * context left usable.  Synchronises `stream`. */
lv_status lv_ctx_selftest_barrier(lv_ctx *ctx, void *stream);

/* Architecture constants (Section 2.1: features proportional to FLOPs and to
 * memory I/O).  With P_layer = d*hq*hd + 2*d*hkv*hd + hq*hd*d + 3*d*F:
 *   phi[0] = 2*L*P_layer/tp       FLOPs per new token
 *   phi[1] = 2*L*hkv*hd*kv_bytes/tp  KV bytes per context token
 *   phi[2] = 2*L*hq*hd/tp         causal-attention FLOPs per p^2
 *   *weight_bytes = L*P_layer*weight_bytes/tp   bytes of weights read per step
 * Host only.  LV_EINVAL for non-positive fields or tp not dividing heads/FFN;
 * LV_EOVERFLOW if a constant exceeds int64. */
lv_status lv_arch_constants(const lv_arch *arch, int64_t phi[3], int64_t *weight_bytes);

/* Per-request and per-batch features (Section 2.1 and the sums of Eq. 1).
 *  req_feat   int64[3][n_req] (SoA) or NULL: p*phi0, c*phi1, p^2*phi2.
 *             A product beyond int64 records LV_EDATA and stores INT64_MAX.
 *  batch_feat int64[5][n_batch] (SoA) or NULL: S1 = sum p, S2 = sum c,
 *             S3 = sum p^2, n, n^2.
 *  batch_seg  uint8[n_batch] or NULL: phase*2 + regime under model->split.
 * arch may be NULL when req_feat is NULL; model may be NULL when batch_seg is
 * NULL.  Integer results are exact. */
lv_status lv_features(lv_ctx *ctx, const lv_arch *arch, const lv_model *model, const lv_batches *b,
                      int64_t *req_feat, int64_t *batch_feat, uint8_t *batch_seg, void *stream);

/* Eq. 1 from precomputed aggregates: T[b] = beta + a1*S1 + a2*S2 + a3*S3 + a4*n^2
 * with the coefficients of segment batch_seg[b]; T = 0 where n = 0.
 * batch_feat int64[5][n_batch] as written by lv_features. */
lv_status lv_batch_latency(lv_ctx *ctx, const lv_model *model, const int64_t *batch_feat,
                           const uint8_t *batch_seg, int64_t n_batch, double *T, void *stream);

/* The fused hot path (Eq. 1 plus the additive shares of Section 2.1): one pass
 * over the request arrays computes every batch's sums, segment and T, each
 * request's share t_i, and (if acc != NULL) adds every share into the tenant
 * accumulator.  T double[n_batch] (or NULL), share double[n_req] (or NULL).
 * b->tenant and b->n_tenants must match acc when acc is given.
 * Arithmetic: on the default path every share is the correctly rounded value of
 * fl(fl(beta/n) + fl(a4*n)) + a1 p + a2 c + a3 p^2 evaluated exactly in integer
 * fixed point, and T the correctly rounded value of Eq. 1 evaluated exactly;
 * results agree with a left-to-right double evaluation to a few ulp. */
lv_status lv_attribute(lv_ctx *ctx, const lv_model *model, const lv_batches *b, double *T, double *share,
                       lv_tenant_acc *acc, void *stream);

/* Single-precision variant of lv_attribute: T and shares evaluated in fp32
 * (coefficients rounded to float; T by Eq. 1 in four fused multiply-adds; a
 * share as fl(beta/n) + fl(a4 n) + p (a1 + a3 p) + a2 c in fused multiply-adds)
 * and written as float (device float[n_batch], float[n_req], either may be
 * NULL).  Within 1e-5 relative of the exact results for this package's
 * workloads (shares relative to max(|share|, T/n)).  With acc, the tenant totals
 * are the exact sums of the fp32 shares (each rounded to 2^-72 s, as
 * lv_attribute's).  Errors as lv_attribute; float outputs 4-byte aligned. */
lv_status lv_attribute_f32(lv_ctx *ctx, const lv_model *model, const lv_batches *b, float *T, float *share,
                           lv_tenant_acc *acc, void *stream);

/* Per-tenant accumulator (Section 2: L_u).  Every fp64 share is rounded to a
 * multiple of 2^-72 s (exact for shares of at least 2^-20 s; the rounding error
 * is below 1.1e-22 s otherwise) and summed EXACTLY in a 128-bit integer per
 * tenant, so totals do not depend on summation order and are bit-identical run
 * to run; lv_tenant_totals returns the correctly rounded fp64 value of each
 * exact sum.  A total beyond +-2^55 s records LV_EDATA.  Accumulation
 * continues across calls until reset. */
lv_status lv_tenant_acc_create(lv_ctx *ctx, int32_t n_tenants, lv_tenant_acc **out);
void lv_tenant_acc_destroy(lv_tenant_acc *acc);
lv_status lv_tenant_acc_reset(lv_tenant_acc *acc, void *stream);
/* Add share[i] to tenant[i]'s total for i < n_req (device arrays). */
lv_status lv_tenant_accumulate(lv_ctx *ctx, lv_tenant_acc *acc, const double *share, const int32_t *tenant,
                               int64_t n_req, void *stream);
/* L double[n_tenants] (device): the current totals. */
lv_status lv_tenant_totals(lv_ctx *ctx, lv_tenant_acc *acc, double *L, void *stream);
/* One serving step (Section 2.1: attribution runs inside the scheduler, once
 * per engine step): lv_attribute of the step's batches, then, with acc, the
 * per-tenant totals, as lv_attribute followed by lv_tenant_totals would give
 * them.  flags: 0 or LV_STEP_RESET, which starts acc from zero before the
 * step's shares are added (the totals are then this step's alone).  L is
 * double[n_tenants] (device) or NULL; L and LV_STEP_RESET need acc.  T, share,
 * acc and the errors are as for lv_attribute; results are bit-identical to the
 * separate calls.  A step of at most 4,096 requests in at most 16 batches,
 * with at most 512 tenants, is one kernel launch (one thread-block cluster);
 * larger inputs run the separate calls' kernels. */
#define LV_STEP_RESET 1
lv_status lv_attribute_step(lv_ctx *ctx, const lv_model *model, const lv_batches *b, double *T, double *share,
                            lv_tenant_acc *acc, double *L, int32_t flags, void *stream);
/* Checkpoint / resume: the exact state is n_tenants * 16 bytes (host buffer).
 * export synchronises the stream. */
int64_t lv_tenant_acc_state_bytes(const lv_tenant_acc *acc);
lv_status lv_tenant_acc_export(lv_tenant_acc *acc, void *host_state, int64_t bytes, void *stream);
lv_status lv_tenant_acc_import(lv_tenant_acc *acc, const void *host_state, int64_t bytes, void *stream);

/* Ordinary least squares of Eq. 1's coefficients per segment (Section 2.1:
 * "fit the coefficients via ordinary least squares on profiling data").
 * y is double[n_y][n_batch] (device): n_y latency vectors for the same batches,
 * fitted in one pass over the requests.  inout[0..n_y-1] are HOST models: their
 * split is read (all must be equal) and their coefficients are overwritten for
 * every group whose status is LV_OK.  rep (host, may be NULL) receives one
 * lv_fit_report per y vector.  Decode batches have p_i = 1, so S1 == S3: when
 * that holds for every batch of a group the a3 column is dropped and a1
 * carries a1 + a3.  Empty batches are skipped.  The Gram matrix is accumulated
 * exactly in integers and X^T y exactly in fixed point (y on a 2^-100 s grid);
 * the solve runs in double-double after power-of-two column scaling.
 * Limits: 1 <= n_y <= 4; batch sums S1, S2, S3 and n^2 below 2^48 (else
 * LV_EOVERFLOW); every y finite with |y| < 2^25 s (else LV_EDATA).  Returns LV_OK
 * once the pass has completed, whatever the groups' outcomes (rep[k].status[g]);
 * models are left untouched on any other return.  Synchronous: returns after
 * the coefficients are on the host, and consumes the context's sticky status
 * (a data error recorded by an earlier asynchronous call is reported here). */
lv_status lv_fit(lv_ctx *ctx, const lv_batches *b, const double *y, int32_t n_y, lv_model *inout,
                 lv_fit_report *rep, void *stream);

/* The token-count baseline the paper compares against (VTC, Tables 1-2): for
 * each of n_y latency vectors y (device double[n_y][n_batch], as lv_fit), one
 * least-squares line T = beta + a * S1 over every non-empty batch, whatever its
 * phase and regime (S1: the batch's total new tokens).  The sums come from the
 * same exact pass as lv_fit; the 2x2 normal equations are solved with an exact
 * integer determinant and double-double numerators.  coef: host
 * double[n_y][2] (beta, a), written where status[k] is LV_OK; status: host
 * int32[n_y] (LV_OK, LV_ENODATA for fewer than 2 batches, LV_ESINGULAR when
 * every batch has the same S1); count: host int64[n_y] (batches used) or NULL.
 * Synchronous.  Errors as lv_fit. */
lv_status lv_fit_vtc(lv_ctx *ctx, const lv_batches *b, const double *y, int32_t n_y, double *coef, int32_t *status,
                     int64_t *count, void *stream);

/* Accuracy of predicted batch latencies T against measured y (both device
 * double[n]; Section 3.2, Tables 1-2), over the batches with y > 0: both forms
 * of R^2, the mean relative error and its nearest-rank p50/p90/p99 (the
 * ceil(q m / 100)-th smallest of the m relative errors, exact; each error is
 * fl(fl(T - y) / y), as fp64 arithmetic gives it).  When every sample's y and
 * non-zero T lie on one grid 2^(E - 78), E the largest binary exponent among
 * them, and -160 <= E <= 224, the sums are exact integers and R^2 is rounded
 * once from them; otherwise (a non-finite value, magnitudes too far apart or
 * extreme) they are fp64 in a fixed order.  The mean relative error is an
 * fp64 sum in a fixed order.  Either way results repeat bit for bit.  n < 2^32
 * (LV_EINVAL otherwise).  One cooperative kernel launch: its blocks meet at
 * grid-wide barriers whose waits are bounded (a few seconds), after which the
 * call returns LV_ETIMEOUT.  rep: host.  With no sample every value is NaN and
 * n = 0; an R^2 whose denominator is 0 is NaN.  Synchronous. */
lv_status lv_accuracy(lv_ctx *ctx, const double *y, const double *T, int64_t n, lv_accuracy_report *rep,
                      void *stream);

/* What-if (Section 1: admission control and what-if planning over alternative
 * batch mixes).  For every pending request j (p_new, c_new, phase_new: device
 * int32[n_pending]) and candidate batch k of `cand`:
 *   T_new[j][k]     = Eq. 1 of the batch cand_k + {j}
 *   share_new[j][k] = request j's share in that batch.
 * Outputs double[n_pending][n_cand] (device, row-major, pending-major); either
 * may be NULL. */
lv_status lv_whatif(lv_ctx *ctx, const lv_model *model, const lv_batches *cand, const int32_t *p_new,
                    const int32_t *c_new, const int32_t *phase_new, int64_t n_pending, double *T_new,
                    double *share_new, void *stream);

/* What-if with admission (Section 1: what-if planning for admission control).
 * lv_whatif's outputs, plus
 *   admit[j][k] = 1 if L[u_j] + share_new[j][k] <= budget[u_j] (one fp64
 *                 addition) and T_new[j][k] <= slo, else 0,
 * with u_j = tenant_new[j] (device int32[n_pending]); L and budget are device
 * double[n_tenants] (L, e.g., from lv_tenant_totals: each tenant's attributed
 * latency so far; budget its allowance), slo in seconds.  admit: device
 * uint8[n_pending][n_cand], required; T_new and share_new may be NULL.  A
 * tenant id outside [0, n_tenants) records LV_EDATA and that request's pairs
 * get 0.  Pointers misaligned for their type, n_tenants <= 0 or a NULL admit,
 * L or budget: LV_EINVAL. */
lv_status lv_whatif_admit(lv_ctx *ctx, const lv_model *model, const lv_batches *cand, const int32_t *p_new,
                          const int32_t *c_new, const int32_t *phase_new, const int32_t *tenant_new,
                          int64_t n_pending, const double *L, const double *budget, int32_t n_tenants, double slo,
                          double *T_new, double *share_new, uint8_t *admit, void *stream);

/* Attribution without any allocation (the paper has no counterpart; this is a
 * service to callers that cannot allocate device memory at call time).  A
 * serving engine typically reserves nearly all GPU memory for its KV cache up
 * front and must not grow its footprint inside the scheduling loop, and a
 * cudaMalloc there would also synchronise the device on the latency-critical
 * path; such a caller cannot create an lv_ctx (which allocates scratch).
 *
 * Computes exactly what lv_attribute computes for T and share (no tenant
 * accumulation), with default arithmetic, using instead of an lv_ctx a fixed
 * scratch area that lives in the library image as a static device array
 * (about 2.6 MB on every GPU that loads the library, held until the process
 * exits).  It calls no cudaMalloc, cudaFree or other allocating routine.
 *  - Limit: n_batch + n_req must not exceed 67,108,864 (65,536 tiles of 1,024
 *    batch boundaries and requests); larger inputs return LV_EINVAL before
 *    anything is launched.
 *  - status: optional DEVICE int32 (caller-owned).  It is set to 0 on the
 *    stream, then kernels OR in 1 for invalid input data (other bits are
 *    reserved); read it after synchronising the stream.
 *  - The first call on each device looks up the scratch array's device address
 *    (cudaGetSymbolAddress) and caches it; make that first call before any
 *    stream capture.
 *  - Every call uses the same scratch array, which keeps the previous call's
 *    contents (each call rewrites what it reads).  Calls whose work overlaps
 *    on the GPU (different streams, or several host threads) race on it:
 *    serialise them.
 * Other arguments and errors as for lv_attribute. */
lv_status lv_attribute_noalloc(const lv_model *model, const lv_batches *b, double *T, double *share,
                               int32_t *status, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* LLMVISOR_H */
