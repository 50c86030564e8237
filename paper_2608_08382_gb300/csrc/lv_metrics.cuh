// Accuracy of predicted batch latencies against measured ones (Section 3.2,
// Tables 1-2: R^2 and percentiles of the relative error), over the samples,
// the batches with y > 0 (m of them):
//   r2_ssr  = 1 - sum (y - T)^2 / sum (y - mean y)^2
//   r2_corr = (sum (y - mean y)(T - mean T))^2 / (sum (y - mean y)^2 sum (T - mean T)^2)
//   rel_b   = |T_b - y_b| / y_b (difference and quotient each rounded to
//             double, as fp64 arithmetic gives them), its mean and its
//             nearest-rank p50, p90, p99 (the ceil(q m / 100)-th smallest).
//
// GB300 issues fp64 at 1/64 of the fp32 rate, so the common case runs on the
// integer pipes, exactly:
//   k_acc_range    the largest binary exponent Emax among the samples' y and
//                  non-zero T, and the exponent of the lowest set bit among
//                  them.  When every such value lies on the grid 2^(Emax - 78)
//                  and Emax is moderate, the exact path below is taken.
//   k_acc_exact    per sample the integers Y = y 2^S and T 2^S (S = 78 - Emax,
//                  both below 2^79 in magnitude) and D = Y - T; the exact sums
//                  of Y, T, Y^2, T^2 and D^2, from which
//                    m sxx = m sum Y^2 - (sum Y)^2,   m syy = m sum T^2 - (sum T)^2,
//                    2 m sxy = m (sum Y^2 + sum T^2 - sum D^2) - 2 sum Y sum T,
//                    m ssr = m sum D^2
//                  follow exactly (all on the grid 2^(-2S), which both R^2
//                  cancel); and rel by exact integer division.
//   k_acc_sums,    otherwise (a non-finite sample value, magnitudes too far
//   k_acc_moments  apart, or extreme ones): the same quantities in fp64, means
//                  first, then centred moments, each in a fixed order.
//   k_acc_select   the percentiles, exact: rel is a non-negative double, so
//                  its bit pattern orders like its value, and a
//                  most-significant-digit radix select (11-bit digits below the
//                  prefix that every sample shares, one shared-memory histogram
//                  per distinct prefix, the digit picked on the device) finds
//                  the bit pattern of the element of each target rank.  The
//                  first pass also sums rel in fixed point anchored at the
//                  largest rel (terms below 2^-100 of it truncated).
// Blocks never wait on one another: each fold runs in the block that finishes
// last (an atomic ticket, reset for the next launch), and every kernel of a
// call runs back to back on the stream with no host round trip.
#pragma once

#include <cstdint>

#include "lv_fit.cuh"

namespace lv {

typedef unsigned __int128 u128;

constexpr int kAccBlock = 256;
constexpr int kAccTargets = 3;  // p50, p90, p99
constexpr int kAccWords = 14;   // per-block partial of the exact sums
constexpr int kAccPart = 16;    // words per block partial (any pass)
constexpr int kSelBits = 11;    // radix digit
constexpr int kSelBins = 1 << kSelBits;
constexpr int kSelBlock = 512;
constexpr int kSelPasses = (63 + kSelBits - 1) / kSelBits;  // a sample's sign bit is 0
constexpr int kAccGrid = 78;  // S = kAccGrid - Emax puts every |v 2^S| below 2^79
// Range of Emax for the exact path: within it the definition's own fp64
// arithmetic (squared deviations, their products in r2_corr) neither overflows
// nor underflows for values on the grid, so the exact results are what fp64
// evaluation approximates.
constexpr int kAccEmaxLo = -160, kAccEmaxHi = 224;
constexpr int kAccLkeyBias = 2100;  // lowest-set-bit exponents stored as kAccLkeyBias - e > 0
constexpr uint64_t kFracMask = (1ull << 52) - 1, kHiddenBit = 1ull << 52;

// Exponent range and exactness of one call (accumulators zero at allocation
// and reset by the block that reads them; the result words are rewritten by
// every call).
struct AccRange {
  int emax;   // max biased exponent of the samples' y and non-zero T
  int lkey;   // max of kAccLkeyBias - (exponent of the lowest set bit)
  int bad;    // a sample's y or T is not finite
  int exact;  // result: the exact path applies
  int S;      // result: grid exponent, S = kAccGrid - Emax
  int pad[3];
};

// Select state: the three prefixes first (they become the percentiles' bit
// patterns and sit right after the eight sums, so one copy reads both).
struct SelState {
  uint64_t pf[kAccTargets];
  int64_t rk[kAccTargets];  // rank still to find below each prefix
  uint64_t relmax;          // largest rel (its bit pattern)
  int shift;                // bits below the settled prefixes; 0 when done
  int pad;
};

// Largest and smallest rel over the samples: max(bits) and max(~bits), so that
// zero is the identity of both (reset by the block that reads them).
struct RelAcc {
  unsigned long long max, nmax;
};

// y > 0 on the bit pattern: sign clear, not zero, not NaN (+inf counts).
__device__ __forceinline__ bool acc_is_sample(uint64_t b) {
  return (int64_t)b > 0 && b <= 0x7FF0000000000000ull;
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

// Sum of `v` over the block in a fixed order (shuffle tree, then the warps in
// index order); the result is valid in thread 0.  `red` holds one double per
// warp.
__device__ __forceinline__ double block_sum_fixed(double v, double *red) {
#pragma unroll
  for (int d = 16; d; d >>= 1) v += __shfl_xor_sync(0xffffffffu, v, d);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  double s = 0.0;
  if (threadIdx.x == 0)
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += red[w];
  return s;
}

// `k` interleaved doubles summed over `blocks` partials with the whole block:
// thread j takes partials j, j + blockDim, ... in order, then the block sum in
// its fixed order; out[0..k) is written by thread 0.
__device__ __forceinline__ void fold_partials(const double *part, int blocks, int k, double *red, double *out) {
  for (int c = 0; c < k; ++c) {
    double s = 0.0;
    for (int b = threadIdx.x; b < blocks; b += blockDim.x) s += __ldcg(part + (int64_t)b * kAccPart + c);
    s = block_sum_fixed(s, red);
    if (threadIdx.x == 0) out[c] = s;
  }
}

__device__ __forceinline__ int block_max_int(int v, int *red) {
  v = (int)__reduce_max_sync(0xffffffffu, (unsigned)v);
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) red[wid] = v;
  __syncthreads();
  int s = 0;
  if (threadIdx.x == 0)
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s = max(s, red[w]);
  return s;  // thread 0
}

__device__ __forceinline__ void range_note(uint64_t b, int &emax, int &lkey, int &bad) {
  const int be = (int)((b >> 52) & 0x7FF);
  if (be == 0x7FF) {
    bad = 1;
    return;
  }
  const uint64_t M = (b & kFracMask) | (be ? kHiddenBit : 0ull);
  const int eb = be ? be : 1;
  emax = max(emax, eb);
  lkey = max(lkey, kAccLkeyBias - (eb - 1075 + __ffsll((long long)M) - 1));
}

// Exponent range of the samples' y and non-zero T, and with it the path.
__global__ void __launch_bounds__(kAccBlock) k_acc_range(const double *__restrict__ y, const double *__restrict__ T,
                                                         int64_t n, AccRange *__restrict__ rg,
                                                         unsigned int *ticket) {
  __shared__ int red[kAccBlock / 32];
  int emax = 0, lkey = 0, bad = 0;
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i < n; i += stride) {
    const uint64_t yb = (uint64_t)__double_as_longlong(__ldg(y + i));
    if (!acc_is_sample(yb)) continue;
    const uint64_t tb = (uint64_t)__double_as_longlong(__ldg(T + i));
    range_note(yb, emax, lkey, bad);
    if (tb << 1) range_note(tb, emax, lkey, bad);
  }
  const int e = block_max_int(emax, red), k = block_max_int(lkey, red), b = block_max_int(bad, red);
  if (threadIdx.x == 0 && e > 0) {
    atomicMax(&rg->emax, e);
    atomicMax(&rg->lkey, k);
    if (b) atomicOr(&rg->bad, 1);
  }
  if (last_block(ticket) && threadIdx.x == 0) {
    const int eb = __ldcg(&rg->emax), lk = __ldcg(&rg->lkey), bd = __ldcg(&rg->bad);
    const int E = eb - 1023, lmin = kAccLkeyBias - lk;
    rg->exact = !bd && n < (int64_t)1 << 32 &&
                (eb == 0 || (E >= kAccEmaxLo && E <= kAccEmaxHi && lmin >= E - kAccGrid));
    rg->S = kAccGrid - E;
    rg->emax = rg->lkey = rg->bad = 0;
  }
}

// ---------------------------------------------------------------- exact path

__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// A quotient digit from its estimate: one below the estimate's integer part
// (never above the true digit when the estimate is within one half of it).
__device__ __forceinline__ uint32_t acc_digit(float e) { return e >= 1.0f ? __float2uint_rz(e) - 1u : 0u; }

// floor(Ma 2^54 / B) for 2^52 <= Ma, B < 2^53 (so the quotient lies in
// [2^53, 2^55)), and whether the remainder is non-zero.  Schoolbook division
// with three digits of 20, 20 and 15 bits: each digit is estimated from a
// single-precision reciprocal of B's top 24 bits (relative error below 2^-21
// all told, so with digits below 2^20 the estimate is within one half of the
// true digit) and settled exactly on the integer remainder, which the digit
// taken one low leaves non-negative and at most two steps away.
__device__ __forceinline__ uint64_t acc_div54(uint64_t Ma, uint64_t B, bool &rem_nz) {
  const float inv = rcp_approx((float)(uint32_t)(B >> 29));  // B >> 29 in [2^23, 2^24): exact in float
  u128 R = (u128)Ma << 54;
  const u128 B35 = (u128)B << 35, B15 = (u128)B << 15;
  uint32_t q1 = acc_digit(__fmul_rn(__ull2float_rn((uint64_t)(R >> 64)), inv));
  R -= ((u128)q1 * B) << 35;
  for (int k = 0; k < 3 && R >= B35; ++k) {
    R -= B35;
    ++q1;
  }
  uint32_t q2 = acc_digit(__fmul_rn(__fmul_rn(__ull2float_rn((uint64_t)(R >> 40)), inv), 0.0625f));
  R -= ((u128)q2 * B) << 15;
  for (int k = 0; k < 3 && R >= B15; ++k) {
    R -= B15;
    ++q2;
  }
  uint32_t q3 = acc_digit(__fmul_rn(__fmul_rn(__ull2float_rn((uint64_t)(R >> 20)), inv), 1.0f / 512.0f));
  R -= (u128)q3 * B;
  for (int k = 0; k < 3 && R >= (u128)B; ++k) {
    R -= B;
    ++q3;
  }
  rem_nz = R != 0;
  return ((uint64_t)q1 << 35) + ((uint64_t)q2 << 15) + q3;
}

// Bit pattern of fl(fl(|D|) / y), where |D| (below 2^80) is |T - y| on the
// grid and y = My 2^ky on the same grid: the difference rounded to 53 bits
// (nearest, ties to even), then the quotient rounded the same way.  Every
// quotient lies in [2^-81, 2^81], a normal double.
__device__ __forceinline__ uint64_t acc_rel_bits(u128 Dm, uint64_t My, int ky) {
  if (Dm == 0) return 0ull;
  const uint64_t dh = (uint64_t)(Dm >> 64), dl = (uint64_t)Dm;
  const int lead = dh ? 127 - __clzll((long long)dh) : 63 - __clzll((long long)dl);
  uint64_t Ma;
  int ka;
  if (lead <= 52) {
    Ma = dl << (52 - lead);
    ka = lead - 52;
  } else {
    int s = lead - 52;  // 1..27: the dropped bits lie in the low word
    Ma = (uint64_t)(Dm >> s);
    const uint64_t low = dl & ((1ull << s) - 1), half = 1ull << (s - 1);
    Ma += (low > half || (low == half && (Ma & 1ull))) ? 1ull : 0ull;
    if (Ma >> 53) {
      Ma >>= 1;
      ++s;
    }
    ka = s;
  }
  bool rem;
  const uint64_t Q = acc_div54(Ma, My, rem);  // rel = (Q + frac) 2^(ka - ky - 54)
  int e = ka - ky - 54;
  uint64_t mant, rb;
  bool st;
  if (Q >> 54) {
    mant = Q >> 2;
    rb = (Q >> 1) & 1ull;
    st = (Q & 1ull) || rem;
    e += 2;
  } else {
    mant = Q >> 1;
    rb = Q & 1ull;
    st = rem;
    e += 1;
  }
  mant += rb & ((st ? 1ull : 0ull) | (mant & 1ull));
  if (mant >> 53) {
    mant >>= 1;
    ++e;
  }
  return ((uint64_t)(e + 1075) << 52) | (mant & kFracMask);
}

__device__ __forceinline__ void add128w(uint64_t *a, u128 x) {
  const u128 s = (((u128)a[1] << 64) | a[0]) + x;
  a[0] = (uint64_t)s;
  a[1] = (uint64_t)(s >> 64);
}

__device__ __forceinline__ void add192w(uint64_t *a, uint64_t w0, uint64_t w1, uint64_t w2) {
  u128 s = (u128)a[0] + w0;
  a[0] = (uint64_t)s;
  s = (u128)a[1] + w1 + (uint64_t)(s >> 64);
  a[1] = (uint64_t)s;
  a[2] += w2 + (uint64_t)(s >> 64);
}

// a += X^2 for X < 2^81 (a: 192 bits).
__device__ __forceinline__ void add_sq(uint64_t *a, u128 X) {
  const uint64_t xl = (uint64_t)X, xh = (uint64_t)(X >> 64);
  const u128 p = (u128)xl * xl, q = (u128)xl * (xh << 1);
  const u128 mid = (p >> 64) + (uint64_t)q;
  add192w(a, (uint64_t)p, (uint64_t)mid, (uint64_t)(q >> 64) + xh * xh + (uint64_t)(mid >> 64));
}

// The exact sums: [0] count, [1..2] sum Y, [3..4] sum T (two's complement),
// [5..7] sum Y^2, [8..10] sum T^2, [11..13] sum D^2.
__device__ __forceinline__ void acc_combine(uint64_t *a, const uint64_t *b) {
  a[0] += b[0];
  add128w(a + 1, ((u128)b[2] << 64) | b[1]);
  add128w(a + 3, ((u128)b[4] << 64) | b[3]);
  add192w(a + 5, b[5], b[6], b[7]);
  add192w(a + 8, b[8], b[9], b[10]);
  add192w(a + 11, b[11], b[12], b[13]);
}

// Block total of the exact sums (integers: any order gives the same result),
// valid in thread 0.  `red`: kAccWords words per warp.
__device__ __forceinline__ void acc_block_combine(uint64_t *w, uint64_t *red) {
#pragma unroll
  for (int d = 16; d; d >>= 1) {
    uint64_t o[kAccWords];
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) o[j] = __shfl_xor_sync(0xffffffffu, w[j], d);
    acc_combine(w, o);
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0)
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) red[wid * kAccWords + j] = w[j];
  __syncthreads();
  if (threadIdx.x == 0)
    for (int v = 1; v < (int)(blockDim.x >> 5); ++v) acc_combine(w, red + v * kAccWords);
}

// One sample on the grid 2^-S (the range pass guarantees both values are
// normal and on it): the sums and rel's bit pattern.
__device__ __forceinline__ uint64_t acc_exact_sample(uint64_t yb, uint64_t tb, int S, uint64_t *w) {
  const uint64_t My = (yb & kFracMask) | kHiddenBit;
  const int ky = (int)(yb >> 52) - 1075 + S;  // y = My 2^ky on the grid, ky <= 26
  const u128 Y = ky >= 0 ? (u128)My << ky : (u128)(My >> min(-ky, 63));
  u128 Tm = 0;
  const bool tneg = (tb >> 63) != 0;
  if (tb << 1) {
    const uint64_t Mt = (tb & kFracMask) | kHiddenBit;
    const int kt = (int)((tb >> 52) & 0x7FF) - 1075 + S;
    Tm = kt >= 0 ? (u128)Mt << kt : (u128)(Mt >> min(-kt, 63));
  }
  w[0] += 1;
  add128w(w + 1, Y);
  add128w(w + 3, tneg ? (u128)0 - Tm : Tm);
  const u128 Dm = tneg ? Y + Tm : (Y >= Tm ? Y - Tm : Tm - Y);
  add_sq(w + 5, Y);
  add_sq(w + 8, Tm);
  add_sq(w + 11, Dm);
  return acc_rel_bits(Dm, My, ky);
}

// 64 x 192 -> 256-bit product.
__device__ __forceinline__ void mul64x192(uint64_t m, const uint64_t *b, uint64_t *w) {
  w[0] = w[1] = w[2] = w[3] = 0;
  acc_add256(w, m * b[0], __umul64hi(m, b[0]), 0, 0);
  acc_add256(w, 0, m * b[1], __umul64hi(m, b[1]), 0);
  acc_add256(w, 0, 0, m * b[2], __umul64hi(m, b[2]));
}

// 128 x 128 -> 256-bit unsigned product.
__device__ __forceinline__ void mul128x128(uint64_t a0, uint64_t a1, uint64_t b0, uint64_t b1, uint64_t *w) {
  w[0] = w[1] = w[2] = w[3] = 0;
  acc_add256(w, a0 * b0, __umul64hi(a0, b0), 0, 0);
  acc_add256(w, 0, a0 * b1, __umul64hi(a0, b1), 0);
  acc_add256(w, 0, a1 * b0, __umul64hi(a1, b0), 0);
  acc_add256(w, 0, 0, a1 * b1, __umul64hi(a1, b1));
}

__device__ __forceinline__ void sub256(uint64_t *a, const uint64_t *b) {
  acc_add256(a, ~b[0], ~b[1], ~b[2], ~b[3]);
  acc_add256(a, 1, 0, 0, 0);
}

// Select state for a new call: the prefix every sample shares (the common
// leading bits of the smallest and largest rel) and the target ranks
// ceil(q m / 100), q = 50, 90, 99.  Resets the rel accumulators.
__device__ __forceinline__ void acc_publish_select(RelAcc *ra, SelState *sel, int64_t m) {
  const uint64_t hi = __ldcg(&ra->max), lo = ~(uint64_t)__ldcg(&ra->nmax);
  ra->max = 0ull;
  ra->nmax = 0ull;
  sel->relmax = hi;
  const int cp = m == 0 || hi == lo ? 64 : __clzll((long long)(hi ^ lo));
  sel->shift = m == 0 ? 0 : 64 - cp;
  const uint64_t pf = cp == 64 ? hi : hi >> (64 - cp);
  for (int t = 0; t < kAccTargets; ++t) {
    const int64_t q = t == 0 ? 50 : t == 1 ? 90 : 99;
    sel->pf[t] = pf;
    sel->rk[t] = (q * m + 99) / 100;
  }
}

__device__ __forceinline__ void acc_note_rel(uint64_t rb, unsigned long long &rmax, unsigned long long &rnmax) {
  rmax = max(rmax, (unsigned long long)rb);
  rnmax = max(rnmax, (unsigned long long)~rb);
}

__device__ __forceinline__ void acc_flush_rel(unsigned long long rmax, unsigned long long rnmax, RelAcc *ra) {
#pragma unroll
  for (int d = 16; d; d >>= 1) {
    rmax = max(rmax, __shfl_xor_sync(0xffffffffu, rmax, d));
    rnmax = max(rnmax, __shfl_xor_sync(0xffffffffu, rnmax, d));
  }
  if ((threadIdx.x & 31) == 0 && (rmax | rnmax)) {
    atomicMax(&ra->max, rmax);
    atomicMax(&ra->nmax, rnmax);
  }
}

// Exact path: the sums and every rel in one pass over y and T; the last block
// folds the block partials and writes sums[0] = m and, scaled by m 2^(2S),
// sums[3..6] = sxx, syy, sxy, ssr.  Returns at once when the range pass chose
// the fp64 path.
__global__ void __launch_bounds__(kAccBlock) k_acc_exact(const double *__restrict__ y, const double *__restrict__ T,
                                                         int64_t n, const AccRange *__restrict__ rg,
                                                         uint64_t *__restrict__ relbits, uint64_t *__restrict__ part,
                                                         double *__restrict__ sums, RelAcc *__restrict__ ra,
                                                         SelState *__restrict__ sel, unsigned int *ticket) {
  __shared__ uint64_t red[kAccBlock / 32 * kAccWords];
  if (!rg->exact) return;
  const int S = rg->S;
  uint64_t w[kAccWords];
#pragma unroll
  for (int j = 0; j < kAccWords; ++j) w[j] = 0ull;
  unsigned long long rmax = 0ull, rnmax = 0ull;
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i < n; i += stride) {
    const uint64_t yb = (uint64_t)__double_as_longlong(__ldg(y + i));
    const uint64_t tb = (uint64_t)__double_as_longlong(__ldg(T + i));
    uint64_t rb = ~0ull;  // not a sample
    if (acc_is_sample(yb)) {
      rb = acc_exact_sample(yb, tb, S, w);
      acc_note_rel(rb, rmax, rnmax);
    }
    relbits[i] = rb;
  }
  acc_flush_rel(rmax, rnmax, ra);
  acc_block_combine(w, red);
  if (threadIdx.x == 0)
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) part[(int64_t)blockIdx.x * kAccPart + j] = w[j];
  if (!last_block(ticket)) return;
#pragma unroll
  for (int j = 0; j < kAccWords; ++j) w[j] = 0ull;
  for (int b = threadIdx.x; b < (int)gridDim.x; b += kAccBlock) {
    uint64_t o[kAccWords];
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) o[j] = __ldcg(part + (int64_t)b * kAccPart + j);
    acc_combine(w, o);
  }
  acc_block_combine(w, red);
  if (threadIdx.x != 0) return;
  const uint64_t m = w[0];
  // |sum T| and its sign
  const bool tneg = (int64_t)w[4] < 0;
  const u128 st = ((u128)w[4] << 64) | w[3], sa = tneg ? (u128)0 - st : st;
  const uint64_t s0 = (uint64_t)sa, s1 = (uint64_t)(sa >> 64);
  uint64_t sxx[4], syy[4], sxy[4], ssr[4], tmp[4];
  mul64x192(m, w + 5, sxx);
  mul128x128(w[1], w[2], w[1], w[2], tmp);
  sub256(sxx, tmp);
  mul64x192(m, w + 8, syy);
  mul128x128(s0, s1, s0, s1, tmp);
  sub256(syy, tmp);
  // 2 m sxy = m (sum Y^2 + sum T^2 - sum D^2) - 2 sum Y sum T; the 192-bit
  // bracket may be negative (two's complement), hence the split below
  uint64_t g[3] = {w[5], w[6], w[7]};
  add192w(g, w[8], w[9], w[10]);
  add192w(g, ~w[11], ~w[12], ~w[13]);
  add192w(g, 1, 0, 0);
  const bool gneg = (int64_t)g[2] < 0;
  if (gneg) {
    g[0] = ~g[0];
    g[1] = ~g[1];
    g[2] = ~g[2];
    add192w(g, 1, 0, 0);
  }
  mul64x192(m, g, sxy);
  if (gneg) {
    uint64_t z[4] = {0, 0, 0, 0};
    sub256(z, sxy);
    sxy[0] = z[0];
    sxy[1] = z[1];
    sxy[2] = z[2];
    sxy[3] = z[3];
  }
  mul128x128(w[1], w[2], s0, s1, tmp);
  acc_add256(tmp, tmp[0], tmp[1], tmp[2], tmp[3]);  // 2 sum Y |sum T|
  if (tneg)
    acc_add256(sxy, tmp[0], tmp[1], tmp[2], tmp[3]);
  else
    sub256(sxy, tmp);
  mul64x192(m, w + 11, ssr);
  sums[0] = (double)m;
  sums[3] = int256_to_dd(sxx, 0).hi;
  sums[4] = int256_to_dd(syy, 0).hi;
  sums[5] = 0.5 * int256_to_dd(sxy, 0).hi;
  sums[6] = int256_to_dd(ssr, 0).hi;
  acc_publish_select(ra, sel, (int64_t)m);
}

// ---------------------------------------------------------------- fp64 path

// Pass 1: per-block count, sum y, sum T over the samples; rel's bit patterns
// stored (all ones for a batch that is not a sample, which the select never
// counts).  The last block folds the partials into sums[0..2] and sets up the
// select.  Returns at once when the range pass chose the exact path.
__global__ void __launch_bounds__(kAccBlock) k_acc_sums(const double *__restrict__ y, const double *__restrict__ T,
                                                        int64_t n, const AccRange *__restrict__ rg,
                                                        uint64_t *__restrict__ relbits, double *__restrict__ part,
                                                        double *__restrict__ sums, RelAcc *__restrict__ ra,
                                                        SelState *__restrict__ sel, unsigned int *ticket) {
  __shared__ double red[kAccBlock / 32];
  if (rg->exact) return;
  double c = 0.0, sy = 0.0, st = 0.0;
  unsigned long long rmax = 0ull, rnmax = 0ull;
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i < n; i += stride) {
    const double yv = y[i], tv = T[i];
    uint64_t bits = ~0ull;
    if (yv > 0.0) {
      c += 1.0;
      sy += yv;
      st += tv;
      bits = (uint64_t)__double_as_longlong(__ddiv_rn(fabs(__dsub_rn(tv, yv)), yv));
      acc_note_rel(bits, rmax, rnmax);
    }
    relbits[i] = bits;
  }
  acc_flush_rel(rmax, rnmax, ra);
  const double a = block_sum_fixed(c, red), b = block_sum_fixed(sy, red), d = block_sum_fixed(st, red);
  if (threadIdx.x == 0) {
    double *p = part + (int64_t)kAccPart * blockIdx.x;
    p[0] = a;
    p[1] = b;
    p[2] = d;
  }
  if (!last_block(ticket)) return;
  fold_partials(part, gridDim.x, 3, red, sums);
  if (threadIdx.x == 0) acc_publish_select(ra, sel, (int64_t)sums[0]);
}

// Pass 2: centred moments with the means from pass 1 (sums = {count, sum y,
// sum T}); the last block folds them into sums[3..6] = sxx, syy, sxy, ssr.
__global__ void __launch_bounds__(kAccBlock) k_acc_moments(const double *__restrict__ y, const double *__restrict__ T,
                                                           int64_t n, const AccRange *__restrict__ rg,
                                                           double *__restrict__ sums, double *__restrict__ part,
                                                           unsigned int *ticket) {
  __shared__ double red[kAccBlock / 32];
  if (rg->exact) return;
  const double m = sums[0];
  const double my = m > 0 ? sums[1] / m : 0.0, mt = m > 0 ? sums[2] / m : 0.0;
  double sxx = 0.0, syy = 0.0, sxy = 0.0, ssr = 0.0;
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i < n; i += stride) {
    const double yv = y[i], tv = T[i];
    if (yv > 0.0) {
      const double dy = yv - my, dt = tv - mt, e = yv - tv;
      sxx += dy * dy;
      syy += dt * dt;
      sxy += dy * dt;
      ssr += e * e;
    }
  }
  const double v0 = block_sum_fixed(sxx, red), v1 = block_sum_fixed(syy, red), v2 = block_sum_fixed(sxy, red),
               v3 = block_sum_fixed(ssr, red);
  if (threadIdx.x == 0) {
    double *p = part + (int64_t)kAccPart * blockIdx.x;
    p[0] = v0;
    p[1] = v1;
    p[2] = v2;
    p[3] = v3;
  }
  if (last_block(ticket)) fold_partials(part, gridDim.x, 4, red, sums + 3);
}

// ---------------------------------------------------------------- percentiles

// rel (bit pattern v, finite, non-negative) on the grid 2^(bemax - 1123),
// bemax the largest rel's biased exponent: below 2^101, truncated under the
// grid (at most 2^-100 of the largest rel per term).
__device__ __forceinline__ u128 acc_rel_fixed(uint64_t v, int bemax) {
  const int be = (int)(v >> 52);
  const uint64_t M = (v & kFracMask) | (be ? kHiddenBit : 0ull);
  const int sv = (be ? be : 1) - bemax + 48;
  return sv >= 0 ? (u128)M << sv : sv > -64 ? (u128)(M >> -sv) : (u128)0;
}

// The three targets' next digit, one warp per target: lane l sums bins
// [64 l, 64 l + 64) of the target's histogram, a warp scan finds the lane
// whose range holds the remaining rank, then the same over that lane's bins
// two at a time.
__device__ __forceinline__ void acc_pick(const unsigned int *__restrict__ hs, SelState *sel, int t, uint64_t pf,
                                         int w) {
  const int lane = threadIdx.x & 31;
  const int64_t r = sel->rk[t];
  const uint4 *h4 = reinterpret_cast<const uint4 *>(hs + 64 * lane);
  uint64_t s = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint4 q = __ldcg(h4 + j);
    s += (uint64_t)q.x + q.y + q.z + q.w;
  }
  uint64_t inc = s;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint64_t o = __shfl_up_sync(0xffffffffu, inc, d);
    if (lane >= d) inc += o;
  }
  unsigned ball = __ballot_sync(0xffffffffu, (int64_t)inc >= r);
  const int L = ball ? __ffs(ball) - 1 : 31;
  const uint64_t below = __shfl_sync(0xffffffffu, inc - s, L);
  const uint2 pr = __ldcg(reinterpret_cast<const uint2 *>(hs + 64 * L) + lane);
  const uint64_t ps = (uint64_t)pr.x + pr.y;
  uint64_t inc2 = ps;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint64_t o = __shfl_up_sync(0xffffffffu, inc2, d);
    if (lane >= d) inc2 += o;
  }
  ball = __ballot_sync(0xffffffffu, (int64_t)(below + inc2) >= r);
  const int L2 = ball ? __ffs(ball) - 1 : 31;
  if (lane == L2) {
    const uint64_t b0 = below + inc2 - ps;
    const bool first = (int64_t)(b0 + pr.x) >= r;
    const int bin = 64 * L + 2 * lane + (first ? 0 : 1);
    sel->rk[t] = r - (int64_t)(first ? b0 : b0 + pr.x);
    sel->pf[t] = (pf << w) | (uint64_t)bin;
  }
}

// One radix-select pass.  Every sample whose bits above `shift` equal a
// target's prefix adds one to that prefix's histogram at its next digit (the
// kSelBits bits below `shift`, fewer at the end); targets with the same
// prefix share one histogram, and prefixes of one length are either equal or
// disjoint, so a sample counts at most once.  The last block picks each
// target's digit and clears the histograms.  Pass 0 also sums rel in fixed
// point into sums[7] (the largest rel itself when it is inf or NaN, which is
// what an exact sum gives then).  Later passes return at once once every
// digit is settled.
__global__ void __launch_bounds__(kSelBlock) k_acc_select(const uint64_t *__restrict__ relbits, int64_t n,
                                                          SelState *__restrict__ sel, unsigned int *__restrict__ hist,
                                                          uint64_t *__restrict__ part, double *__restrict__ sums,
                                                          unsigned int *ticket, int pass) {
  __shared__ unsigned int h[kAccTargets * kSelBins];
  __shared__ uint64_t red[kSelBlock / 32 * 3];
  const int shift = sel->shift;
  const uint64_t relmax = sel->relmax;
  const bool digit = shift > 0;
  const bool rsum = pass == 0 && relmax < 0x7FF0000000000000ull;
  if (!digit && pass != 0) return;
  const uint64_t pf0 = sel->pf[0], pf1 = sel->pf[1], pf2 = sel->pf[2];
  const int w = min(kSelBits, shift), lo = shift - w;
  const uint64_t dmask = (1ull << w) - 1;
  if (digit) {
    for (int i = threadIdx.x; i < kAccTargets * kSelBins; i += kSelBlock) h[i] = 0u;
    __syncthreads();
  }
  const int bemax = max((int)(relmax >> 52), 1);
  uint64_t s0 = 0, s1 = 0, s2 = 0;  // sum of rel on its grid, 192 bits
  const int64_t stride = (int64_t)gridDim.x * kSelBlock;
  for (int64_t i = blockIdx.x * (int64_t)kSelBlock + threadIdx.x; i < n; i += stride) {
    const uint64_t v = __ldcg(relbits + i);
    if (v == ~0ull) continue;  // not a sample
    if (digit) {
      const uint64_t key = v >> shift;
      const int s = key == pf0 ? 0 : key == pf1 ? 1 : key == pf2 ? 2 : -1;
      if (s >= 0) atomicAdd(&h[s * kSelBins + (int)((v >> lo) & dmask)], 1u);
    }
    if (rsum) {
      uint64_t a[3] = {s0, s1, s2};
      const u128 x = acc_rel_fixed(v, bemax);
      add192w(a, (uint64_t)x, (uint64_t)(x >> 64), 0);
      s0 = a[0];
      s1 = a[1];
      s2 = a[2];
    }
  }
  if (digit) {
    __syncthreads();
    for (int i = threadIdx.x; i < kAccTargets * kSelBins; i += kSelBlock) {
      const unsigned int c = h[i];
      if (c) atomicAdd(hist + i, c);
    }
  }
  if (pass == 0) {
    uint64_t a[3] = {s0, s1, s2};
#pragma unroll
    for (int d = 16; d; d >>= 1) {
      const uint64_t o0 = __shfl_xor_sync(0xffffffffu, a[0], d), o1 = __shfl_xor_sync(0xffffffffu, a[1], d),
                     o2 = __shfl_xor_sync(0xffffffffu, a[2], d);
      add192w(a, o0, o1, o2);
    }
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
      red[3 * wid] = a[0];
      red[3 * wid + 1] = a[1];
      red[3 * wid + 2] = a[2];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int v = 1; v < kSelBlock / 32; ++v) add192w(a, red[3 * v], red[3 * v + 1], red[3 * v + 2]);
      uint64_t *p = part + (int64_t)kAccPart * blockIdx.x;
      p[0] = a[0];
      p[1] = a[1];
      p[2] = a[2];
    }
  }
  if (!last_block(ticket)) return;
  if (pass == 0) {
    uint64_t a[3] = {0, 0, 0};
    for (int b = threadIdx.x; b < (int)gridDim.x; b += kSelBlock) {
      const uint64_t *p = part + (int64_t)kAccPart * b;
      add192w(a, __ldcg(p), __ldcg(p + 1), __ldcg(p + 2));
    }
#pragma unroll
    for (int d = 16; d; d >>= 1) {
      const uint64_t o0 = __shfl_xor_sync(0xffffffffu, a[0], d), o1 = __shfl_xor_sync(0xffffffffu, a[1], d),
                     o2 = __shfl_xor_sync(0xffffffffu, a[2], d);
      add192w(a, o0, o1, o2);
    }
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) {
      red[3 * wid] = a[0];
      red[3 * wid + 1] = a[1];
      red[3 * wid + 2] = a[2];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      for (int v = 1; v < kSelBlock / 32; ++v) add192w(a, red[3 * v], red[3 * v + 1], red[3 * v + 2]);
      const uint64_t wv[4] = {a[0], a[1], a[2], 0ull};
      sums[7] = rsum ? ldexp(int256_to_dd(wv, 0).hi, bemax - 1123) : __longlong_as_double((long long)relmax);
    }
  }
  if (!digit) return;
  const int wid = threadIdx.x >> 5;
  if (wid < kAccTargets) {
    const uint64_t pf = wid == 0 ? pf0 : wid == 1 ? pf1 : pf2;
    const int slot = pf == pf0 ? 0 : pf == pf1 ? 1 : 2;
    acc_pick(hist + slot * kSelBins, sel, wid, pf, w);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kAccTargets * kSelBins; i += kSelBlock) hist[i] = 0u;
  if (threadIdx.x == 0) sel->shift = lo;
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
