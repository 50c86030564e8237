// Accuracy of predicted batch latencies against measured ones (Section 3.2,
// Tables 1-2: R^2 and percentiles of the relative error), over the batches
// with y > 0:
//   r2_ssr  = 1 - sum (y - T)^2 / sum (y - mean y)^2
//   r2_corr = (sum (y - mean y)(T - mean T))^2 / (sum (y - mean y)^2 sum (T - mean T)^2)
//   rel_b   = |T_b - y_b| / y_b, its mean and its nearest-rank p50, p90, p99
//             (the ceil(q m)-th smallest of the m values).
// Sums are fp64 in a fixed order (per-thread strided sums, a fixed shuffle
// tree per block, then the block partials in index order), so results repeat
// bit for bit.  The percentiles are exact: rel is a non-negative double, so its
// bit pattern orders like its value, and a most-significant-digit radix select
// (8 bits per pass, one shared-memory histogram per block, the digit chosen on
// the device) finds the bit pattern of the element of each target rank.
#pragma once

#include <cstdint>

#include "lv_fit.cuh"

namespace lv {

constexpr int kAccBlock = 256;
constexpr int kAccBins = 256;  // one 8-bit digit per pass
constexpr int kAccTargets = 3;  // p50, p90, p99

__device__ __forceinline__ double block_sum_fixed(double v, double *red) {
#pragma unroll
  for (int d = 16; d; d >>= 1) v += __shfl_xor_sync(0xffffffffu, v, d);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0)
    for (int w = 0; w < kAccBlock / 32; ++w) s += red[w];
  return s;  // thread 0
}

// True in the block that finishes last (its partial and every other block's
// are visible to it then).  The ticket is reset for the next launch; blocks
// never wait on one another.
__device__ __forceinline__ bool last_block(unsigned int *ticket) {
  __shared__ bool last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    last = atomicAdd(ticket, 1u) == gridDim.x - 1;
    if (last) *ticket = 0u;
  }
  __syncthreads();
  if (last) __threadfence();
  return last;
}

// `k` interleaved values summed over `blocks` partials, in index order.
__device__ __forceinline__ void fold_partials(const double *part, int blocks, int k, double *out) {
  if (threadIdx.x < k) {
    double s = 0.0;
    for (int b = 0; b < blocks; ++b) s += part[(int64_t)b * k + threadIdx.x];
    out[threadIdx.x] = s;
  }
}

// Pass 1: per-block count, sum y, sum T over y > 0; rel's bit patterns stored
// (all ones for y <= 0, which the select never counts).  The last block folds
// the partials into tot[0..2].
__global__ void __launch_bounds__(kAccBlock) k_acc_sums(const double *__restrict__ y, const double *__restrict__ T,
                                                        int64_t n, uint64_t *__restrict__ relbits,
                                                        double *__restrict__ part, double *__restrict__ tot,
                                                        unsigned int *ticket) {
  __shared__ double red[kAccBlock / 32];
  double c = 0.0, sy = 0.0, st = 0.0;
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i < n; i += stride) {
    const double yv = y[i], tv = T[i];
    uint64_t bits = ~0ull;
    if (yv > 0.0) {
      c += 1.0;
      sy += yv;
      st += tv;
      bits = (uint64_t)__double_as_longlong(__ddiv_rn(fabs(__dsub_rn(tv, yv)), yv));
    }
    relbits[i] = bits;
  }
  const double a = block_sum_fixed(c, red), b = block_sum_fixed(sy, red), d = block_sum_fixed(st, red);
  if (threadIdx.x == 0) {
    part[3 * blockIdx.x] = a;
    part[3 * blockIdx.x + 1] = b;
    part[3 * blockIdx.x + 2] = d;
  }
  if (last_block(ticket)) fold_partials(part, gridDim.x, 3, tot);
}

// Pass 2: centred moments with the means from pass 1 (tot = {count, sum y,
// sum T}); the last block folds them into tot[3..7].
__global__ void __launch_bounds__(kAccBlock) k_acc_moments(const double *__restrict__ y, const double *__restrict__ T,
                                                           const uint64_t *__restrict__ relbits, int64_t n,
                                                           double *__restrict__ tot, double *__restrict__ part,
                                                           unsigned int *ticket) {
  __shared__ double red[kAccBlock / 32];
  const double m = tot[0];
  const double my = m > 0 ? tot[1] / m : 0.0, mt = m > 0 ? tot[2] / m : 0.0;
  double sxx = 0.0, syy = 0.0, sxy = 0.0, ssr = 0.0, srel = 0.0;
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i < n; i += stride) {
    const double yv = y[i], tv = T[i];
    if (yv > 0.0) {
      const double dy = yv - my, dt = tv - mt, e = yv - tv;
      sxx += dy * dy;
      syy += dt * dt;
      sxy += dy * dt;
      ssr += e * e;
      srel += __longlong_as_double((long long)relbits[i]);
    }
  }
  const double v0 = block_sum_fixed(sxx, red), v1 = block_sum_fixed(syy, red), v2 = block_sum_fixed(sxy, red),
               v3 = block_sum_fixed(ssr, red), v4 = block_sum_fixed(srel, red);
  if (threadIdx.x == 0) {
    double *p = part + 5 * blockIdx.x;
    p[0] = v0;
    p[1] = v1;
    p[2] = v2;
    p[3] = v3;
    p[4] = v4;
  }
  if (last_block(ticket)) fold_partials(part, gridDim.x, 5, tot + 3);
}

// After a histogram pass: for each target, the digit whose bin holds its rank
// (ranks ceil(q m / 100), q = 50, 90, 99, set from the sample count m at the
// first pass), appended to its prefix; the histograms are cleared for the next
// pass.  One warp: lane t < 3 takes target t.  All passes run back to back on
// the stream with no host round trip.
__device__ __forceinline__ void acc_pick(unsigned int *__restrict__ hist, const double *__restrict__ sums,
                                         uint64_t *__restrict__ prefix, int64_t *__restrict__ rank, int pass) {
  const int t = threadIdx.x;
  if (t < kAccTargets) {
    int64_t r;
    uint64_t pf;
    if (pass == 0) {
      const int64_t m = (int64_t)sums[0];
      const int64_t q = t == 0 ? 50 : t == 1 ? 90 : 99;
      r = (q * m + 99) / 100;
      pf = 0;
    } else {
      r = rank[t];
      pf = prefix[t];
    }
    int64_t below = 0;
    int d = 0;
    for (; d < kAccBins - 1; ++d) {
      const unsigned int c = hist[t * kAccBins + d];
      if (below + c >= r) break;
      below += c;
    }
    rank[t] = r - below;
    prefix[t] = (pf << 8) | (uint64_t)d;
  }
  __syncwarp();
  for (int i = t; i < kAccTargets * kAccBins; i += 32) hist[i] = 0u;
}

// One radix-select pass: for each target t whose top `shift`..63 bits are
// prefix[t] (shift = 64 - 8 * passes done), count the next 8-bit digit; the
// last block picks each target's digit and clears the histograms.
__global__ void __launch_bounds__(kAccBlock) k_acc_hist(const uint64_t *__restrict__ relbits, int64_t n,
                                                        uint64_t *__restrict__ prefix, int shift,
                                                        unsigned int *__restrict__ hist, const double *__restrict__ sums,
                                                        int64_t *__restrict__ rank, unsigned int *ticket) {
  __shared__ unsigned int h[kAccTargets][kAccBins];
  for (int i = threadIdx.x; i < kAccTargets * kAccBins; i += kAccBlock) (&h[0][0])[i] = 0u;
  __syncthreads();
  uint64_t pf[kAccTargets];
#pragma unroll
  for (int t = 0; t < kAccTargets; ++t) pf[t] = prefix[t];
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i < n; i += stride) {
    const uint64_t v = relbits[i];
    if (v == ~0ull) continue;  // y <= 0: not a sample
    const unsigned int dig = (unsigned int)(v >> (shift - 8)) & 0xffu;
#pragma unroll
    for (int t = 0; t < kAccTargets; ++t) {
      const bool match = shift == 64 || (v >> shift) == pf[t];
      if (match) atomicAdd(&h[t][dig], 1u);
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kAccTargets * kAccBins; i += kAccBlock) {
    const unsigned int c = (&h[0][0])[i];
    if (c) atomicAdd(hist + i, c);
  }
  if (last_block(ticket) && threadIdx.x < 32) acc_pick(hist, sums, prefix, rank, (64 - shift) / 8);
}

// After a histogram pass: for each target, the digit whose bin holds its rank
// (ranks ceil(q m / 100), q = 50, 90, 99, set from the sample count m at the
// first pass), appended to its prefix; the histograms are cleared for the next
// pass.  One warp: lane t < 3 takes target t.  All passes then run back to back
// on the stream with no host round trip.
__global__ void __launch_bounds__(32) k_acc_pick(unsigned int *__restrict__ hist, const double *__restrict__ sums,
                                                 uint64_t *__restrict__ prefix, int64_t *__restrict__ rank, int pass) {
  const int t = threadIdx.x;
  if (t < kAccTargets) {
    int64_t r;
    uint64_t pf;
    if (pass == 0) {
      const int64_t m = (int64_t)sums[0];
      const int64_t q = t == 0 ? 50 : t == 1 ? 90 : 99;
      r = (q * m + 99) / 100;
      pf = 0;
    } else {
      r = rank[t];
      pf = prefix[t];
    }
    int64_t below = 0;
    int d = 0;
    for (; d < kAccBins - 1; ++d) {
      const unsigned int c = hist[t * kAccBins + d];
      if (below + c >= r) break;
      below += c;
    }
    rank[t] = r - below;
    prefix[t] = (pf << 8) | (uint64_t)d;
  }
  __syncwarp();
  for (int i = t; i < kAccTargets * kAccBins; i += 32) hist[i] = 0u;
}

// ---------------------------------------------------------------- token-count baseline
//
// The token-count baseline (VTC, compared against in Tables 1-2): one line
// T = beta + a S1 over every non-empty batch, whatever its phase and regime.
// Its normal equations are sums the fit pass already forms exactly: the Gram
// entries (1,1), (1,S1), (S1,S1) and the X^T y entries of the columns 1 and S1,
// added over the four groups.  The determinant n sum S1^2 - (sum S1)^2 is formed
// exactly in integers (0 exactly when every batch has the same S1: singular);
// the numerators and the division in double-double.

struct VtcOut {
  double beta, a;
  int64_t n;
  int32_t status, pad;
};

// 128 x 128 -> 256-bit unsigned product.
__device__ __forceinline__ void mul128x128(uint64_t a0, uint64_t a1, uint64_t b0, uint64_t b1, uint64_t *w) {
  w[0] = w[1] = w[2] = w[3] = 0;
  acc_add256(w, a0 * b0, __umul64hi(a0, b0), 0, 0);
  acc_add256(w, 0, a0 * b1, __umul64hi(a0, b1), 0);
  acc_add256(w, 0, a1 * b0, __umul64hi(a1, b0), 0);
  acc_add256(w, 0, 0, a1 * b1, __umul64hi(a1, b1));
}

__global__ void __launch_bounds__(32) k_vtc_solve(const FitAcc *__restrict__ totals, int n_y, VtcOut *__restrict__ out) {
  const int k = threadIdx.x;
  if (k >= n_y) return;
  const int NE = fit_entries(n_y);
  uint64_t g00[4] = {0, 0, 0, 0}, g01[4] = {0, 0, 0, 0}, g11[4] = {0, 0, 0, 0}, r0[4] = {0, 0, 0, 0},
           r1[4] = {0, 0, 0, 0};
  for (int g = 0; g < 4; ++g) {
    const FitAcc *T = totals + g * NE;
    const uint64_t *a = T[gram_idx(0, 0)].w, *b = T[gram_idx(0, 1)].w, *c = T[gram_idx(1, 1)].w;
    const uint64_t *d = T[15 + k * 5].w, *e = T[15 + k * 5 + 1].w;
    acc_add256(g00, a[0], a[1], a[2], a[3]);
    acc_add256(g01, b[0], b[1], b[2], b[3]);
    acc_add256(g11, c[0], c[1], c[2], c[3]);
    acc_add256(r0, d[0], d[1], d[2], d[3]);
    acc_add256(r1, e[0], e[1], e[2], e[3]);
  }
  VtcOut o{0.0, 0.0, (int64_t)g00[0], LV_OK, 0};
  if (o.n < 2) {
    o.status = LV_ENODATA;
    out[k] = o;
    return;
  }
  // det = n * sum S1^2 - (sum S1)^2, exact (n < 2^63, both sums below 2^128)
  uint64_t p[4], q[4];
  mul128x128(g00[0], 0, g11[0], g11[1], p);
  mul128x128(g01[0], g01[1], g01[0], g01[1], q);
  uint64_t det[4] = {p[0], p[1], p[2], p[3]};
  acc_add256(det, ~q[0], ~q[1], ~q[2], ~q[3]);
  acc_add256(det, 1, 0, 0, 0);  // p - q, two's complement
  if ((det[0] | det[1] | det[2] | det[3]) == 0) {
    o.status = LV_ESINGULAR;
    out[k] = o;
    return;
  }
  const dd D = int256_to_dd(det, 0), G00 = int256_to_dd(g00, 0), G01 = int256_to_dd(g01, 0),
           G11 = int256_to_dd(g11, 0), R0 = int256_to_dd(r0, kFitYLsb), R1 = int256_to_dd(r1, kFitYLsb);
  const dd beta = dd_div(dd_add(dd_mul(G11, R0), dd_neg(dd_mul(G01, R1))), D);
  const dd slope = dd_div(dd_add(dd_mul(G00, R1), dd_neg(dd_mul(G01, R0))), D);
  o.beta = beta.hi + beta.lo;
  o.a = slope.hi + slope.lo;
  out[k] = o;
}

}  // namespace lv
