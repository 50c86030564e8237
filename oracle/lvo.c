/*
 * LLMVisor CPU oracle -- TEST INFRASTRUCTURE, NOT PART OF THE PRODUCT.
 *
 * A plain, slow, obviously correct restatement of the attribution model of
 * "LLMVisor: A Real-Time Latency Attribution Model for Multi-Tenant LLM
 * Serving": per-request features, per-batch reduction, the piecewise-linear
 * batch latency of Eq. 1, additive per-request shares, per-tenant roll-up and
 * what-if evaluation.  Only tests/, __graft_entry__.smoke() and bench.py's CPU
 * baseline leg may load it.  It shares no code, header or table with the CUDA
 * library under paper_2608_08382_gb300/.
 *
 * Everything is double precision evaluated strictly left to right; compile with
 * -ffp-contract=off so no multiply-add is fused.  Inputs are trusted (the
 * callers are tests); there is no validation beyond overflow of int64 products.
 *
 * Readings of the paper taken here (where it is silent or ambiguous):
 *  - Eq. 1's last term  a4 * sum_i |B|  is taken literally as a4 * n^2.
 *  - A batch's phase is prefill if any of its requests is a prefill, else decode.
 *  - The regime is compute-bound when S1 = sum_i p_i >= split[phase], else
 *    memory-bound.
 *  - Each request's share is  beta/n + a1 p_i + a2 c_i + a3 p_i^2 + a4 n :
 *    the fixed cost and the n^2 term are split equally, slope terms go to the
 *    request that carries the feature.
 *  - An empty batch has T = 0, segment (decode, memory) and no shares.
 *
 * Coefficients are double[4][5] indexed [phase * 2 + regime][beta, a1, a2, a3, a4].
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>

#define LVO_OK 0
#define LVO_EINVAL (-1)
#define LVO_EOVERFLOW (-2)

static int mul64(int64_t a, int64_t b, int64_t *out) { return __builtin_mul_overflow(a, b, out) ? 1 : 0; }
static int add64(int64_t a, int64_t b, int64_t *out) { return __builtin_add_overflow(a, b, out) ? 1 : 0; }

/*
 * Architecture constants (Section 2.1: features "proportional to FLOPs and I/O
 * traffic"; the paper fits the proportionality instead of deriving it, so these
 * only rescale feature columns).  Dense transformer, gated FFN with three
 * matrices, biases, embeddings and LM head ignored, weights sharded over tp:
 *   P_layer = d*(hq*hd) + 2*d*(hkv*hd) + (hq*hd)*d + 3*d*F      parameters/layer
 *   phi1 = 2*L*P_layer/tp          FLOPs per new token (GEMMs)
 *   phi2 = 2*L*hkv*hd*kvb/tp       KV-cache bytes loaded per context token
 *   phi3 = 2*L*hq*hd/tp            causal-attention FLOPs per p^2
 *   W    = L*P_layer*wb/tp         weight bytes loaded per step (the beta term)
 * arch = {L, d, hq, hkv, hd, F, wb, kvb, tp}.  tp must divide hq, hkv and F.
 */
int lvo_arch_constants(const int32_t *arch, int64_t *phi, int64_t *w_bytes)
{
    int64_t L = arch[0], d = arch[1], hq = arch[2], hkv = arch[3], hd = arch[4];
    int64_t F = arch[5], wb = arch[6], kvb = arch[7], tp = arch[8];
    for (int k = 0; k < 9; ++k)
        if (arch[k] <= 0) return LVO_EINVAL;
    if (hq % tp || hkv % tp || F % tp) return LVO_EINVAL;
    int64_t q, kv, t1, t2, t3, t4, P;
    int ovf = 0;
    ovf |= mul64(hq, hd, &q);
    ovf |= mul64(hkv, hd, &kv);
    ovf |= mul64(d, q, &t1);          /* Q projection  */
    ovf |= mul64(2 * d, kv, &t2);     /* K and V projections */
    ovf |= mul64(q, d, &t3);          /* output projection */
    ovf |= mul64(3 * d, F, &t4);      /* gate, up, down */
    ovf |= add64(t1, t2, &P);
    ovf |= add64(P, t3, &P);
    ovf |= add64(P, t4, &P);
    int64_t a, b;
    ovf |= mul64(2 * L, P, &a);
    phi[0] = a / tp;
    ovf |= mul64(2 * L, kv, &a);
    ovf |= mul64(a, kvb, &b);
    phi[1] = b / tp;
    ovf |= mul64(2 * L, q, &a);
    phi[2] = a / tp;
    ovf |= mul64(L, P, &a);
    ovf |= mul64(a, wb, &b);
    *w_bytes = b / tp;
    return ovf ? LVO_EOVERFLOW : LVO_OK;
}

/*
 * Per-request physical features (Section 2.1): p_i*phi1 FLOPs, c_i*phi2 bytes,
 * p_i^2*phi3 FLOPs.  out is int64[3][n] (struct of arrays).
 */
int lvo_request_features(int64_t n, const int32_t *p, const int32_t *c, const int64_t *phi, int64_t *out)
{
    int ovf = 0;
    for (int64_t i = 0; i < n; ++i) {
        int64_t pi = p[i], ci = c[i], pp = pi * pi, v;
        ovf |= mul64(pi, phi[0], &v);
        out[i] = v;
        ovf |= mul64(ci, phi[1], &v);
        out[n + i] = v;
        ovf |= mul64(pp, phi[2], &v);
        out[2 * n + i] = v;
    }
    return ovf ? LVO_EOVERFLOW : LVO_OK;
}

/*
 * One batch's reduction (Eq. 1 sums) and segment.
 * feat = {S1 = sum p, S2 = sum c, S3 = sum p^2, n, n^2}; returns the segment
 * code phase*2 + regime.
 */
static int batch_reduce(const int32_t *p, const int32_t *c, const int32_t *phase, int64_t lo, int64_t hi,
                        const int64_t *split, int64_t feat[5])
{
    int64_t S1 = 0, S2 = 0, S3 = 0;
    int prefill = 0;
    for (int64_t i = lo; i < hi; ++i) {
        S1 += p[i];
        S2 += c[i];
        S3 += (int64_t)p[i] * (int64_t)p[i];
        if (phase[i] == 1) prefill = 1;
    }
    int64_t n = hi - lo;
    feat[0] = S1;
    feat[1] = S2;
    feat[2] = S3;
    feat[3] = n;
    feat[4] = n * n;
    if (n == 0) return 0;
    int regime = S1 >= split[prefill] ? 1 : 0;
    return prefill * 2 + regime;
}

/* Batch aggregates for every batch: feat int64[5][n_batch] (SoA), seg uint8[n_batch]. */
void lvo_batch_features(int64_t n_batch, const int64_t *off, const int32_t *p, const int32_t *c,
                        const int32_t *phase, const int64_t *split, int64_t *feat, uint8_t *seg)
{
    for (int64_t b = 0; b < n_batch; ++b) {
        int64_t f[5];
        int s = batch_reduce(p, c, phase, off[b], off[b + 1], split, f);
        for (int k = 0; k < 5; ++k) feat[k * n_batch + b] = f[k];
        seg[b] = (uint8_t)s;
    }
}

/* Eq. 1: T = beta + a1*S1 + a2*S2 + a3*S3 + a4*n^2, left to right. */
static double eq1(const double *k, const int64_t f[5])
{
    if (f[3] == 0) return 0.0;
    double T = k[0];
    T = T + k[1] * (double)f[0];
    T = T + k[2] * (double)f[1];
    T = T + k[3] * (double)f[2];
    T = T + k[4] * (double)f[4];
    return T;
}

/* Eq. 1 from precomputed aggregates (feat SoA [5][n_batch], seg). */
void lvo_batch_latency(int64_t n_batch, const int64_t *feat, const uint8_t *seg, const double *coef, double *T)
{
    for (int64_t b = 0; b < n_batch; ++b) {
        int64_t f[5];
        for (int k = 0; k < 5; ++k) f[k] = feat[k * n_batch + b];
        T[b] = eq1(coef + 5 * seg[b], f);
    }
}

/*
 * Additive per-request share (Section 2.1, "closed-form, additive per-request
 * attributions via Eq. 1"; problem formulation of Section 2: shares sum to the
 * batch latency):  t_i = beta/n + a1 p_i + a2 c_i + a3 p_i^2 + a4 n.
 */
static double share_of(const double *k, int64_t n, int64_t pi, int64_t ci)
{
    double t = k[0] / (double)n;
    t = t + k[1] * (double)pi;
    t = t + k[2] * (double)ci;
    t = t + k[3] * (double)(pi * pi);
    t = t + k[4] * (double)n;
    return t;
}

/* T (may be NULL) per batch and share per request. */
void lvo_attribute(int64_t n_batch, const int64_t *off, const int32_t *p, const int32_t *c,
                   const int32_t *phase, const int64_t *split, const double *coef, double *T, double *share)
{
    for (int64_t b = 0; b < n_batch; ++b) {
        int64_t f[5];
        int s = batch_reduce(p, c, phase, off[b], off[b + 1], split, f);
        const double *k = coef + 5 * s;
        if (T) T[b] = eq1(k, f);
        for (int64_t i = off[b]; i < off[b + 1]; ++i) share[i] = share_of(k, f[3], p[i], c[i]);
    }
}

/*
 * Per-tenant usage L_u = sum over requests of tenant u of their shares
 * (Section 2, problem formulation).  Summed in request order with Neumaier's
 * compensated summation; (sum, comp) carry the running state across calls and
 * L_u = sum_u + comp_u.
 */
void lvo_tenant_accumulate(int64_t n, const double *share, const int32_t *tenant, double *sum, double *comp)
{
    for (int64_t i = 0; i < n; ++i) {
        int32_t u = tenant[i];
        double x = share[i], s = sum[u], t = s + x;
        if (fabs(s) >= fabs(x))
            comp[u] += (s - t) + x;
        else
            comp[u] += (x - t) + s;
        sum[u] = t;
    }
}

void lvo_tenant_totals(int32_t n_tenants, const double *sum, const double *comp, double *L)
{
    for (int32_t u = 0; u < n_tenants; ++u) L[u] = sum[u] + comp[u];
}

/*
 * What-if (Section 1: admission and "what-if" planning over alternative batch
 * mixes).  For every pending request j and candidate batch b the batch
 * B' = B_b + {j} is materialised (j appended last) and evaluated like any other
 * batch: T_new[j][b] = T(B'), share_new[j][b] = share of j in B'.
 */
void lvo_whatif(int64_t n_cand, const int64_t *off, const int32_t *p, const int32_t *c, const int32_t *phase,
                int64_t n_pend, const int32_t *p_new, const int32_t *c_new, const int32_t *phase_new,
                const int64_t *split, const double *coef, double *T_new, double *share_new)
{
    int64_t maxn = 0;
    for (int64_t b = 0; b < n_cand; ++b)
        if (off[b + 1] - off[b] > maxn) maxn = off[b + 1] - off[b];
    int32_t *bp = (int32_t *)malloc(sizeof(int32_t) * (size_t)(maxn + 1));
    int32_t *bc = (int32_t *)malloc(sizeof(int32_t) * (size_t)(maxn + 1));
    int32_t *bph = (int32_t *)malloc(sizeof(int32_t) * (size_t)(maxn + 1));
    for (int64_t j = 0; j < n_pend; ++j) {
        for (int64_t b = 0; b < n_cand; ++b) {
            int64_t n0 = off[b + 1] - off[b];
            memcpy(bp, p + off[b], sizeof(int32_t) * (size_t)n0);
            memcpy(bc, c + off[b], sizeof(int32_t) * (size_t)n0);
            memcpy(bph, phase + off[b], sizeof(int32_t) * (size_t)n0);
            bp[n0] = p_new[j];
            bc[n0] = c_new[j];
            bph[n0] = phase_new[j];
            int64_t f[5];
            int s = batch_reduce(bp, bc, bph, 0, n0 + 1, split, f);
            const double *k = coef + 5 * s;
            T_new[j * n_cand + b] = eq1(k, f);
            share_new[j * n_cand + b] = share_of(k, f[3], bp[n0], bc[n0]);
        }
    }
    free(bp);
    free(bc);
    free(bph);
}
