// Least-squares fit of Eq. 1's coefficients (Section 2.1: "ordinary least
// squares on profiling data", one coefficient set per phase and regime).
//
// For every group g (segment phase*2 + regime) the design rows are the batch
// sums x = [1, S1, S2, S3, n^2] of the profiled batches of that group and the
// targets are their measured latencies y.  The normal equations need the Gram
// matrix X^T X and X^T y per group.  Both are accumulated EXACTLY:
//   - X^T X in 128-bit integers (features are integers below 2^48, so each
//     product is below 2^96);
//   - X^T y in 256-bit fixed point with y rounded to a multiple of 2^-100 s
//     (exact for any latency whose lowest bit is at least 2^-100 s).
// The tile kernel computes the batch sums anyway; in fit mode each of the
// (group, entry) accumulators is owned by one thread of the CTA, which adds the
// contributions of the tile's batches of its group in registers.  CTA partials
// are reduced exactly (integer adds) and each group's small system is solved in
// double-double (about 106-bit) arithmetic after power-of-two column scaling,
// by Cholesky, with singular and under-determined groups reported.
#pragma once

#include "lv_kernels.cuh"

namespace lv {

// ---------------------------------------------------------------- reduction across CTAs

// totals[ge] = sum over CTAs of partial[cta][ge]: one block per entry, threads
// striding over the CTAs, then a tree in shared memory.  Integer addition is
// associative, so the exact result does not depend on the order; the flag
// entries are ORed.
constexpr int kFitRedThreads = 256;
__global__ void __launch_bounds__(kFitRedThreads) k_fit_reduce(const FitAcc *__restrict__ partial, int n_cta,
                                                               int n_ent, FitAcc *__restrict__ totals) {
  __shared__ FitAcc red[kFitRedThreads];
  const int ge = blockIdx.x;
  const bool is_flag = ge % (n_ent / 4) == n_ent / 4 - 1;
  FitAcc t;
  t.w[0] = t.w[1] = t.w[2] = t.w[3] = 0;
  for (int c = threadIdx.x; c < n_cta; c += kFitRedThreads) {
    const FitAcc p = partial[(int64_t)c * n_ent + ge];
    if (is_flag)
      t.w[0] |= p.w[0];
    else
      acc_add256(t.w, p.w[0], p.w[1], p.w[2], p.w[3]);
  }
  red[threadIdx.x] = t;
  __syncthreads();
  for (int h = kFitRedThreads / 2; h > 0; h >>= 1) {
    if ((int)threadIdx.x < h) {
      const FitAcc o = red[threadIdx.x + h];
      if (is_flag)
        red[threadIdx.x].w[0] |= o.w[0];
      else
        acc_add256(red[threadIdx.x].w, o.w[0], o.w[1], o.w[2], o.w[3]);
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) totals[ge] = red[0];
}

// ---------------------------------------------------------------- double-double arithmetic
// Error-free transformations (Knuth's two-sum, Dekker's product via FMA) and the
// usual double-double operations built on them.

struct dd {
  double hi, lo;
};

__device__ __forceinline__ dd two_sum(double a, double b) {
  const double s = __dadd_rn(a, b);
  const double bb = __dsub_rn(s, a);
  const double e = __dadd_rn(__dsub_rn(a, __dsub_rn(s, bb)), __dsub_rn(b, bb));
  return dd{s, e};
}

__device__ __forceinline__ dd quick_two_sum(double a, double b) {
  const double s = __dadd_rn(a, b);
  return dd{s, __dsub_rn(b, __dsub_rn(s, a))};
}

__device__ __forceinline__ dd dd_add(dd x, dd y) {
  dd s = two_sum(x.hi, y.hi);
  const dd t = two_sum(x.lo, y.lo);
  s.lo = __dadd_rn(s.lo, t.hi);
  s = quick_two_sum(s.hi, s.lo);
  s.lo = __dadd_rn(s.lo, t.lo);
  return quick_two_sum(s.hi, s.lo);
}

__device__ __forceinline__ dd dd_neg(dd x) { return dd{-x.hi, -x.lo}; }

__device__ __forceinline__ dd dd_mul(dd x, dd y) {
  const double p = __dmul_rn(x.hi, y.hi);
  double e = __fma_rn(x.hi, y.hi, -p);
  e = __fma_rn(x.hi, y.lo, e);
  e = __fma_rn(x.lo, y.hi, e);
  return quick_two_sum(p, e);
}

__device__ __forceinline__ dd dd_div(dd x, dd y) {
  const double q1 = __ddiv_rn(x.hi, y.hi);
  dd r = dd_add(x, dd_neg(dd_mul(dd{q1, 0.0}, y)));
  const double q2 = __ddiv_rn(r.hi, y.hi);
  r = dd_add(r, dd_neg(dd_mul(dd{q2, 0.0}, y)));
  const double q3 = __ddiv_rn(r.hi, y.hi);
  dd q = quick_two_sum(q1, q2);
  return dd_add(q, dd{q3, 0.0});
}

__device__ __forceinline__ dd dd_scale(dd x, int e) { return dd{ldexp(x.hi, e), ldexp(x.lo, e)}; }

// Signed 256-bit integer (w, two's complement) times 2^E as double-double.
// The leading 123 bits form a window whose value is below 2^123, so its
// rounding to double (at most 2^123) converts back to fixed point without
// overflow; hi is that rounding and lo the correctly rounded exact remainder.
// Bits below the window are dropped (relative 2^-122).
__device__ __forceinline__ dd int256_to_dd(const uint64_t *w, int E) {
  uint64_t v[4] = {w[0], w[1], w[2], w[3]};
  const bool neg = (int64_t)v[3] < 0;
  if (neg) {
    for (int i = 0; i < 4; ++i) v[i] = ~v[i];
    for (int i = 0; i < 4; ++i) {
      if (++v[i] != 0) break;
    }
  }
  int top = 3;
  while (top > 0 && v[top] == 0) --top;
  if (v[top] == 0) return dd{0.0, 0.0};
  const int L = 64 * top + 63 - __clzll((long long)v[top]);  // leading bit
  i128 win;
  int Ew = E;
  if (L <= 122) {
    win = mk128(v[0], v[1]);
  } else {
    const int sh = L - 122;  // right shift that puts the leading bit on bit 122
    const int q = sh >> 6, rb = sh & 63;
    const uint64_t a0 = v[q], a1 = q + 1 < 4 ? v[q + 1] : 0, a2 = q + 2 < 4 ? v[q + 2] : 0;
    win.lo = rb ? (a0 >> rb) | (a1 << (64 - rb)) : a0;
    win.hi = rb ? (a1 >> rb) | (a2 << (64 - rb)) : a1;
    Ew = E + sh;
  }
  const double hi = fix_to_double(win, Ew).d;
  bool ovf = false;
  const i128 back = double_to_fix(hi, Ew, &ovf);
  const double lo = fix_to_double(add128(win, neg128(back)), Ew).d;
  const dd r{hi, lo};
  return neg ? dd_neg(r) : r;
}

struct FitOut {
  double coef[5];
  double ssr, r2;
  int64_t n;
  int32_t status, dropped;
};

// Index of Gram pair (a, b) in the accumulator order (row-major upper triangle).
__host__ __device__ constexpr int gram_idx(int a, int b) {
  return a <= b ? a * 5 - a * (a - 1) / 2 + (b - a) : b * 5 - b * (b - 1) / 2 + (a - b);
}

// Row and column of Gram entry e (inverse of gram_idx: a <= b, row order).
__device__ __forceinline__ void gram_ab(int e, int &a, int &b) {
  a = 0;
  while (e >= 5 - a) {
    e -= 5 - a;
    ++a;
  }
  b = a + e;
}

__device__ __forceinline__ dd dd_sub(dd x, dd y) { return dd_add(x, dd_neg(y)); }

// One warp per (y vector k, group g), block k * 4 + g: builds, scales and
// solves the normal equations from the exact totals.  Lanes convert the 21
// totals at once; the Cholesky factorisation goes column by column, the pivot
// on one lane and the rest of the column on the lanes of its rows; the
// substitutions run on lane 0; the residual sum of squares adds its 30 terms
// on 30 lanes.  A dropped a3 column becomes a unit row and column with a zero
// right-hand side (its coefficient solves to 0).  Each pivot is inverted once
// in double-double and the eliminations multiply.  Loops stay rolled: the
// kernel runs once per fit, so its code is fetched cold.
__global__ void __launch_bounds__(32) k_fit_solve(const FitAcc *__restrict__ totals, int n_y, FitOut *__restrict__ out) {
  __shared__ dd G[15], R[5], L[15], rs[5], inv[5], zz[5];
  __shared__ dd YY;
  __shared__ double cf[5];
  __shared__ int sc[5], sing;
  const int lane = threadIdx.x;
  const int k = blockIdx.x / 4, g = blockIdx.x % 4;
  if (k >= n_y) return;
  const int NE = fit_entries(n_y);
  const FitAcc *T = totals + g * NE;
  FitOut o;
  for (int i = 0; i < 5; ++i) o.coef[i] = 0.0;
  o.ssr = 0.0;
  o.r2 = 0.0;
  o.dropped = 0;
  const int64_t n = (int64_t)T[0].w[0];  // Gram (0,0) = number of batches
  o.n = n;
  const bool drop3 = n > 0 && (T[NE - 1].w[0] & 1ull) == 0ull;
  if (drop3) o.dropped = 1 << 3;
  if (n < (drop3 ? 4 : 5)) {
    o.status = LV_ENODATA;
    if (lane == 0) out[k * 4 + g] = o;
    return;
  }
  // exact totals as double-double, one per lane
  if (lane < 15)
    G[lane] = int256_to_dd(T[lane].w, 0);
  else if (lane < 20)
    R[lane - 15] = int256_to_dd(T[15 + k * 5 + (lane - 15)].w, kFitYLsb);
  else if (lane == 20)
    YY = int256_to_dd(T[15 + 5 * n_y + k].w, kFitYYLsb);
  if (lane == 0) sing = 0;
  __syncwarp();
  if (drop3 && lane < 5) G[gram_idx(lane, 3)] = dd{lane == 3 ? 1.0 : 0.0, 0.0};
  if (drop3 && lane == 5) R[3] = dd{0.0, 0.0};
  __syncwarp();
  // power-of-two column scaling: scaled diagonal near 1
  if (lane < 5) {
    int ex;
    frexp(G[gram_idx(lane, lane)].hi, &ex);
    sc[lane] = -(ex / 2);
  }
  __syncwarp();
  if (lane < 15) {
    int a, b;
    gram_ab(lane, a, b);
    L[lane] = dd_scale(G[lane], sc[a] + sc[b]);
  } else if (lane < 20) {
    rs[lane - 15] = dd_scale(R[lane - 15], sc[lane - 15]);
  }
  __syncwarp();
  // Cholesky G = L L^T (lower triangle in L, indexed symmetrically)
  for (int j = 0; j < 5; ++j) {
    if (lane == j) {
      dd d = L[gram_idx(j, j)];
      for (int m = 0; m < j; ++m) d = dd_sub(d, dd_mul(L[gram_idx(j, m)], L[gram_idx(j, m)]));
      if (!(d.hi > 1e-24)) {
        sing = 1;
      } else {
        // square root in double-double: s0 = sqrt(d.hi) and one Newton step, whose
        // correction needs only a double factor 1/(2 s0); the inverse by one
        // Newton step from the double reciprocal r0 = 1/s0
        const double s0 = sqrt(d.hi), r0 = 1.0 / s0;
        const dd s0sq = dd_mul(dd{s0, 0.0}, dd{s0, 0.0});
        const dd s = dd_add(dd{s0, 0.0}, dd_mul(dd_sub(d, s0sq), dd{0.5 * r0, 0.0}));
        L[gram_idx(j, j)] = s;
        const dd e = dd_sub(dd{1.0, 0.0}, dd_mul(s, dd{r0, 0.0}));
        inv[j] = dd_add(dd{r0, 0.0}, dd_mul(dd{r0, 0.0}, e));
      }
    }
    __syncwarp();
    if (sing) {
      o.status = LV_ESINGULAR;
      if (lane == 0) out[k * 4 + g] = o;
      return;
    }
    if (lane > j && lane < 5) {
      dd v = L[gram_idx(lane, j)];
      for (int m = 0; m < j; ++m) v = dd_sub(v, dd_mul(L[gram_idx(lane, m)], L[gram_idx(j, m)]));
      L[gram_idx(lane, j)] = dd_mul(v, inv[j]);
    }
    __syncwarp();
  }
  if (lane == 0) {
    for (int i = 0; i < 5; ++i) {
      dd v = rs[i];
      for (int m = 0; m < i; ++m) v = dd_sub(v, dd_mul(L[gram_idx(i, m)], zz[m]));
      zz[i] = dd_mul(v, inv[i]);
    }
    for (int i = 4; i >= 0; --i) {
      dd v = zz[i];
      for (int m = i + 1; m < 5; ++m) v = dd_sub(v, dd_mul(L[gram_idx(m, i)], zz[m]));
      zz[i] = dd_mul(v, inv[i]);  // the solution overwrites z, highest index first
      cf[i] = (drop3 && i == 3) ? 0.0 : ldexp(zz[i].hi + zz[i].lo, sc[i]);
    }
  }
  __syncwarp();
  for (int i = 0; i < 5; ++i) o.coef[i] = cf[i];
  // residuals of the rounded coefficients: SSR = y'y - 2 c'X'y + c'Gc (unscaled),
  // one term per lane, summed across the warp
  dd term{0.0, 0.0};
  if (lane < 25) {
    const int i = lane / 5, j = lane % 5;
    term = dd_mul(dd_mul(dd{cf[i], 0.0}, dd{cf[j], 0.0}), G[gram_idx(i, j)]);
  } else if (lane < 30) {
    term = dd_neg(dd_scale(dd_mul(dd{cf[lane - 25], 0.0}, R[lane - 25]), 1));
  }
#pragma unroll
  for (int d = 16; d; d >>= 1)
    term = dd_add(term, dd{__shfl_xor_sync(0xffffffffu, term.hi, d), __shfl_xor_sync(0xffffffffu, term.lo, d)});
  if (lane == 0) {
    const dd sy = R[0];
    const dd ssr = dd_add(YY, term);
    const dd sst = dd_sub(YY, dd_div(dd_mul(sy, sy), dd{(double)n, 0.0}));
    o.ssr = ssr.hi + ssr.lo;
    const double sstv = sst.hi + sst.lo;
    o.r2 = sstv != 0.0 ? 1.0 - o.ssr / sstv : __longlong_as_double(0x7ff8000000000000ll);
    o.status = LV_OK;
    out[k * 4 + g] = o;
  }
}

}  // namespace lv
