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

// totals[ge] = sum over CTAs of partial[cta][ge] (exact integer adds; the flag entry is ORed).
__global__ void k_fit_reduce(const FitAcc *__restrict__ partial, int n_cta, int n_ent, FitAcc *__restrict__ totals) {
  const int ge = blockIdx.x * blockDim.x + threadIdx.x;
  if (ge >= n_ent) return;
  FitAcc t;
  t.w[0] = t.w[1] = t.w[2] = t.w[3] = 0;
  const int e = ge % (n_ent / 4);
  const bool is_flag = e == n_ent / 4 - 1;
  for (int c = 0; c < n_cta; ++c) {
    const FitAcc &p = partial[(int64_t)c * n_ent + ge];
    if (is_flag)
      t.w[0] |= p.w[0];
    else
      acc_add256(t.w, p.w[0], p.w[1], p.w[2], p.w[3]);
  }
  totals[ge] = t;
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

// One thread per (y vector, group): builds, scales and solves the normal
// equations from the exact totals.
__global__ void k_fit_solve(const FitAcc *__restrict__ totals, int n_y, FitOut *__restrict__ out) {
  const int t = threadIdx.x;
  if (t >= 4 * n_y) return;
  const int k = t / 4, g = t % 4;
  const int NE = fit_entries(n_y);
  const FitAcc *T = totals + g * NE;
  FitOut o;
  for (int i = 0; i < 5; ++i) o.coef[i] = 0.0;
  o.ssr = 0.0;
  o.r2 = 0.0;
  o.dropped = 0;
  const int64_t n = (int64_t)T[0].w[0];  // Gram (0,0) = number of batches
  o.n = n;
  const bool any_ne = (T[NE - 1].w[0] & 1ull) != 0;
  int cols[5], kc = 0;
  for (int a = 0; a < 5; ++a) {
    if (a == 3 && n > 0 && !any_ne) {
      o.dropped |= 1 << 3;
      continue;
    }
    cols[kc++] = a;
  }
  if (n < kc) {
    o.status = LV_ENODATA;
    out[k * 4 + g] = o;
    return;
  }
  // Gram in double-double; index of pair (a, b), a <= b
  auto gidx = [](int a, int b) {
    if (a > b) {
      const int tt = a;
      a = b;
      b = tt;
    }
    return a * 5 - a * (a - 1) / 2 + (b - a);
  };
  dd G[5][5], r[5];
  int sc[5];
  for (int i = 0; i < kc; ++i) {
    const FitAcc &d = T[gidx(cols[i], cols[i])];
    const dd gii = int256_to_dd(d.w, 0);
    int ex;
    frexp(gii.hi, &ex);
    sc[i] = -(ex / 2);  // column scale 2^sc, makes the scaled diagonal ~1
  }
  for (int i = 0; i < kc; ++i) {
    for (int j = 0; j < kc; ++j) G[i][j] = dd_scale(int256_to_dd(T[gidx(cols[i], cols[j])].w, 0), sc[i] + sc[j]);
    r[i] = dd_scale(int256_to_dd(T[15 + k * 5 + cols[i]].w, kFitYLsb), sc[i]);
  }
  // Cholesky G = L L^T (in place, lower triangle)
  for (int j = 0; j < kc; ++j) {
    dd d = G[j][j];
    for (int m = 0; m < j; ++m) d = dd_add(d, dd_neg(dd_mul(G[j][m], G[j][m])));
    if (!(d.hi > 1e-24)) {
      o.status = LV_ESINGULAR;
      out[k * 4 + g] = o;
      return;
    }
    // square root in double-double: s0 = sqrt(d.hi), one Newton step
    const double s0 = sqrt(d.hi);
    const dd s0sq = dd_mul(dd{s0, 0.0}, dd{s0, 0.0});
    const dd corr = dd_div(dd_add(d, dd_neg(s0sq)), dd{2.0 * s0, 0.0});
    const dd s = dd_add(dd{s0, 0.0}, corr);
    G[j][j] = s;
    for (int i = j + 1; i < kc; ++i) {
      dd v = G[i][j];
      for (int m = 0; m < j; ++m) v = dd_add(v, dd_neg(dd_mul(G[i][m], G[j][m])));
      G[i][j] = dd_div(v, s);
    }
  }
  dd z[5], a[5];
  for (int i = 0; i < kc; ++i) {
    dd v = r[i];
    for (int m = 0; m < i; ++m) v = dd_add(v, dd_neg(dd_mul(G[i][m], z[m])));
    z[i] = dd_div(v, G[i][i]);
  }
  for (int i = kc - 1; i >= 0; --i) {
    dd v = z[i];
    for (int m = i + 1; m < kc; ++m) v = dd_add(v, dd_neg(dd_mul(G[m][i], a[m])));
    a[i] = dd_div(v, G[i][i]);
  }
  for (int i = 0; i < kc; ++i) o.coef[cols[i]] = ldexp(a[i].hi + a[i].lo, sc[i]);
  // residuals of the rounded coefficients: SSR = y'y - 2 c'X'y + c'Gc (unscaled)
  dd cxy{0.0, 0.0}, cgc{0.0, 0.0}, sy = int256_to_dd(T[15 + k * 5 + 0].w, kFitYLsb);
  for (int i = 0; i < kc; ++i) {
    const dd ci{o.coef[cols[i]], 0.0};
    cxy = dd_add(cxy, dd_mul(ci, int256_to_dd(T[15 + k * 5 + cols[i]].w, kFitYLsb)));
    for (int j = 0; j < kc; ++j)
      cgc = dd_add(cgc, dd_mul(dd_mul(ci, dd{o.coef[cols[j]], 0.0}), int256_to_dd(T[gidx(cols[i], cols[j])].w, 0)));
  }
  const dd yy = int256_to_dd(T[15 + 5 * n_y + k].w, kFitYYLsb);
  const dd ssr = dd_add(dd_add(yy, dd_neg(dd_scale(cxy, 1))), cgc);
  const dd sst = dd_add(yy, dd_neg(dd_div(dd_mul(sy, sy), dd{(double)n, 0.0})));
  o.ssr = ssr.hi + ssr.lo;
  const double sstv = sst.hi + sst.lo;
  o.r2 = sstv != 0.0 ? 1.0 - o.ssr / sstv : __longlong_as_double(0x7ff8000000000000ll);
  o.status = LV_OK;
  out[k * 4 + g] = o;
}

}  // namespace lv
