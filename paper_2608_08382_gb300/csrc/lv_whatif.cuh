// What-if evaluation over (pending request x candidate batch) pairs (Section 1:
// "what-if" planning over alternative batch mixes, admission control).
//
// For candidate batch b with sums (S1, S2, S3, n) and pending request j with
// (p, c), the batch b + {j} has sums (S1 + p, S2 + c, S3 + p^2, n + 1) and its
// phase is prefill if either side is.  With s the segment of b + {j}, Eq. 1 and
// j's share regroup as
//     T  = [beta + a1 S1 + a2 S2 + a3 S3 + a4 (n+1)^2]  +  [a1 p + a2 c + a3 p^2]
//        =            U_b[s]                            +         V_j[s]
//     t_j = [fl(beta/(n+1)) + fl(a4 (n+1))]             +         V_j[s]
//        =            W_b[s]                            +         V_j[s]
// U, W and V are exact 128-bit fixed-point values, precomputed for all four
// segments, so every pair costs a segment select, two exact additions and two
// roundings.  In fp64 mode (or outside the exact range) a pair is evaluated
// left to right in double like any other batch.
#pragma once

#include "lv_kernels.cuh"
#include "lv_warp.cuh"

namespace lv {

struct CandP {
  i128 U[4];
  i128 W[4];
  int64_t s1, s2, s3, n;
  int32_t prefill;
  int32_t slow;  // 1: evaluate pairs of this candidate in fp64
};

struct PendP {
  i128 V[4];
  int32_t p, c, phase, slow;
  double Lu, Bu;  // admission: the request's tenant's running total and budget
};

// Admission inputs (null: plain what-if).  A pair (j, b) is admissible when
// L[u_j] + share_new[j][b] <= budget[u_j] (one fp64 addition) and
// T_new[j][b] <= slo (Section 1: what-if planning for admission control).
struct AdmitArgs {
  const int32_t *tenant;  // [n_pending]
  const double *L, *budget;  // [n_tenants]
  int32_t n_tenants;
  double slo;
  uint8_t *admit;  // [n_pending][n_cand]
};

// Per candidate: U_b[s], W_b[s] for every segment, from the batch sums.
__global__ void k_wi_cand(ModelP mp, const int64_t *__restrict__ bfeat, const uint8_t *__restrict__ bseg,
                          int64_t nc, CandP *__restrict__ out) {
  const int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (b >= nc) return;
  CandP cp;
  cp.s1 = bfeat[b];
  cp.s2 = bfeat[nc + b];
  cp.s3 = bfeat[2 * nc + b];
  cp.n = bfeat[3 * nc + b];
  cp.prefill = (bseg[b] >> 1) & 1;
  cp.slow = mp.fixed ? 0 : 1;
  const int64_t n1 = cp.n + 1;
  const uint64_t F4 = (uint64_t)n1 * (uint64_t)n1;
#pragma unroll
  for (int s = 0; s < 4; ++s) {
    cp.U[s] = mk128(0, 0);
    cp.W[s] = mk128(0, 0);
    if (!mp.fixed) continue;
    const SegFix &f = mp.fx[s];
    if ((uint64_t)cp.s1 > f.lim[0] || (uint64_t)cp.s2 > f.lim[1] || (uint64_t)cp.s3 > f.lim[2] || F4 > f.lim[3] ||
        n1 > 0x7fffffffll) {
      cp.slow = 1;
      continue;
    }
    i128 U = f.B;
    U = add128(U, mul128_u64(f.A1, (uint64_t)cp.s1));
    U = add128(U, mul128_u64(f.A2, (uint64_t)cp.s2));
    U = add128(U, mul128_u64(f.A3, (uint64_t)cp.s3));
    U = add128(U, mul128_u64(f.A4, F4));
    cp.U[s] = U;
    bool slow = false;
    cp.W[s] = batch_k(mp, s, n1, &slow).kf;
    if (slow) cp.slow = 1;
  }
  out[b] = cp;
}

// Per pending request: V_j[s] = a1 p + a2 c + a3 p^2 for every segment.
// With admission, also the request's tenant's total and budget (a tenant id
// out of range records a data error and makes every pair of the request
// inadmissible: NaN compares false).
__global__ void k_wi_pend(ModelP mp, const int32_t *__restrict__ p_new, const int32_t *__restrict__ c_new,
                          const int32_t *__restrict__ ph_new, int64_t np, PendP *__restrict__ out, AdmitArgs adm,
                          int *status) {
  const int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  if (j >= np) return;
  int32_t p = p_new[j], c = c_new[j], ph = ph_new[j];
  int bad = 0;
  check_req(p, c, ph, &bad);
  PendP q;
  q.p = p;
  q.c = c;
  q.phase = ph;
  q.slow = (!mp.fixed || p > kPMaxFix) ? 1 : 0;
  q.Lu = q.Bu = 0.0;
  if (adm.admit) {
    const int32_t u = adm.tenant[j];
    if (u < 0 || u >= adm.n_tenants) {
      bad = 1;
      q.Lu = __longlong_as_double(0x7ff8000000000000ll);
    } else {
      q.Lu = adm.L[u];
      q.Bu = adm.budget[u];
    }
  }
  if (bad) flag(status, kStatusData);
#pragma unroll
  for (int s = 0; s < 4; ++s) {
    q.V[s] = mk128(0, 0);
    if (q.slow) continue;
    const SegFix &f = mp.fx[s];
    const i128 r = add128(f.A1, mul128_u32(f.A3, (uint32_t)p));
    i128 V = mul128_u32(r, (uint32_t)p);
    V = add128(V, f.a2_narrow ? mul_u64_u32(f.A2.lo, (uint32_t)c) : mul128_u32(f.A2, (uint32_t)c));
    q.V[s] = V;
  }
  out[j] = q;
}

// V * 2^E rounded to double: the leading-word rounding for the common
// magnitude 2^64 <= V < 2^96, the general rounding otherwise.
__device__ __forceinline__ double round_fix(i128 V, int E) {
  const uint32_t v3 = (uint32_t)(V.hi >> 32), v2 = (uint32_t)V.hi;
  if (v3 == 0u && v2 != 0u) {
    uint64_t m;
    int ex2;
    return round96((uint32_t)V.lo, (uint32_t)(V.lo >> 32), v2, E, m, ex2);
  }
  return fix_to_double(V, E).d;
}

// Left-to-right fp64 evaluation of one pair (fp64 mode, or outside the exact range).
__device__ __noinline__ void wi_pair_slow(const ModelP &mp, int s, int64_t s1, int64_t s2, int64_t s3, int64_t n1,
                                          int32_t p, int32_t c, double *T, double *share) {
  const BatchAgg g{s1, s2, s3, n1, 1};
  *T = eq1_fp64(mp.coef[s], g);
  bool dummy = false;
  const KEntry e = batch_k(mp, s, n1, &dummy);
  *share = share_fp64(mp.coef[s], e.q, e.a4n, p, c);
}

constexpr int kWiCols = 128;  // candidates per block (one per thread)
constexpr int kWiRows = 32;   // pending requests per block

// Pair grid: block (bx, by) covers candidates [bx*kWiCols, +kWiCols) and pending
// rows [j0 + by*kWiRows, +kWiRows); consecutive threads write consecutive
// candidates of a row, so the row-major [pending][candidate] outputs are
// coalesced.
__global__ void __launch_bounds__(kWiCols) k_wi_pairs(ModelP mp, const CandP *__restrict__ cand,
                                                       const PendP *__restrict__ pend, int64_t nc, int64_t np,
                                                       int64_t j_base, double *__restrict__ T_new,
                                                       double *__restrict__ share_new, double slo,
                                                       uint8_t *__restrict__ admit) {
  static_assert(kWiRows <= kWiCols, "one pending row per thread at most");
  __shared__ PendP sp[kWiRows];
  __shared__ int sE[4];
  const int64_t b = blockIdx.x * (int64_t)kWiCols + threadIdx.x;
  const int64_t j0 = j_base + blockIdx.y * (int64_t)kWiRows;
  const int rows = (int)(np - j0 < kWiRows ? np - j0 : kWiRows);
  int rslow = 0;
  if (threadIdx.x < rows) {
    sp[threadIdx.x] = pend[j0 + threadIdx.x];
    rslow = sp[threadIdx.x].slow;
  }
  if (threadIdx.x < 4) sE[threadIdx.x] = mp.fx[threadIdx.x].E;
  rslow = __syncthreads_or(rslow);
  if (b >= nc) return;
  const CandP *cb = cand + b;
  const int64_t s1 = cb->s1, s2 = cb->s2, s3 = cb->s3, n1 = cb->n + 1;
  const int prefill = cb->prefill, cslow = cb->slow;
  const int64_t sp0 = mp.split[0], sp1 = mp.split[1];
  if (!cslow && !rslow && rows == kWiRows) {
    // every pair of the block exact: no out-of-line call, rows unrolled for
    // independent loads and roundings in flight
#pragma unroll 4
    for (int r = 0; r < kWiRows; ++r) {
      const int32_t p = sp[r].p;
      const int phase = (prefill | sp[r].phase) ? 1 : 0;
      const int s = phase * 2 + ((s1 + p >= (phase ? sp1 : sp0)) ? 1 : 0);
      const i128 V = sp[r].V[s];
      const double T = round_fix(add128(cb->U[s], V), sE[s]);
      const double sh = round_fix(add128(cb->W[s], V), sE[s]);
      const int64_t o = (j0 + r) * nc + b;
      if (T_new) __stcs(T_new + o, T);
      if (share_new) __stcs(share_new + o, sh);
      if (admit) admit[o] = (__dadd_rn(sp[r].Lu, sh) <= sp[r].Bu && T <= slo) ? 1 : 0;
    }
    return;
  }
  for (int r = 0; r < rows; ++r) {
    const int32_t p = sp[r].p, c = sp[r].c;
    const int phase = (prefill | sp[r].phase) ? 1 : 0;
    const int s = phase * 2 + ((s1 + p >= (phase ? sp1 : sp0)) ? 1 : 0);
    double T, sh;
    if (cslow | sp[r].slow) {
      wi_pair_slow(mp, s, s1 + p, s2 + c, s3 + (int64_t)p * p, n1, p, c, &T, &sh);
    } else {
      const i128 V = sp[r].V[s];
      T = round_fix(add128(cb->U[s], V), sE[s]);
      sh = round_fix(add128(cb->W[s], V), sE[s]);
    }
    const int64_t o = (j0 + r) * nc + b;
    if (T_new) __stcs(T_new + o, T);
    if (share_new) __stcs(share_new + o, sh);
    if (admit) admit[o] = (__dadd_rn(sp[r].Lu, sh) <= sp[r].Bu && T <= slo) ? 1 : 0;
  }
}

}  // namespace lv
