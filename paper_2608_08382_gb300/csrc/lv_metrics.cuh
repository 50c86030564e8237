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
//   k_acc_range    the largest and smallest binary exponents Emax, Emin among
//                  the samples' y and non-zero T.  When Emax is finite and
//                  moderate the exact path below is taken: on the grid
//                  2^(Emax - 62) in 64-bit integers when Emax - Emin <= 10 (every
//                  value then lies on it), else on 2^(Emax - 78) in 128-bit
//                  integers, handing over to the fp64 path when a value turns
//                  out not to lie on that grid.
//   k_acc_exact    per sample the integers Y = y 2^S and T 2^S (below 2^63 or
//                  2^79 in magnitude) and D = Y - T; the exact sums
//                  of Y, T, Y^2, T^2 and D^2, from which
//                    m sxx = m sum Y^2 - (sum Y)^2,   m syy = m sum T^2 - (sum T)^2,
//                    2 m sxy = m (sum Y^2 + sum T^2 - sum D^2) - 2 sum Y sum T,
//                    m ssr = m sum D^2
//                  follow exactly (all on the grid 2^(-2S), which both R^2
//                  cancel); and rel by exact integer division.
//   k_acc_sums,    otherwise (a non-finite sample value, extreme magnitudes,
//   k_acc_moments  or a value off the grid): the same quantities in fp64,
//                  means first, then centred moments, each in a fixed order.
//   k_acc_sel0,    the percentiles, exact: rel is a non-negative double, so
//   k_acc_selB,    its bit pattern orders like its value, and a
//   k_acc_sel1,    most-significant-digit radix select finds the bit pattern of
//   k_acc_sel2     the element of each target rank.  The first digit (11 bits
//                  below the prefix every sample shares) is histogrammed over
//                  all samples, which also sums rel in fixed point anchored at
//                  the largest rel (terms below 2^-100 of it truncated); the
//                  next digit over the samples in a target's bin (typically
//                  well under 1% of them); the samples in each target's
//                  second-digit bin (typically a handful) are gathered into a
//                  candidate list, and one block per target settles the
//                  remaining digits on its list.
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
constexpr int kSelFinish = 1024;     // threads of a finishing block (one per target)
constexpr int kSelSmemList = 20480;  // candidates a finishing block holds in shared memory
constexpr int kAccGrid = 78;  // S = kAccGrid - Emax puts every |v 2^S| below 2^79
// Range of Emax for the exact path: within it the definition's own fp64
// arithmetic (squared deviations, their products in r2_corr) neither overflows
// nor underflows for values on the grid, so the exact results are what fp64
// evaluation approximates.
constexpr int kAccEmaxLo = -160, kAccEmaxHi = 224;
constexpr uint64_t kFracMask = (1ull << 52) - 1, kHiddenBit = 1ull << 52;

// Path of one call, rewritten by every call: set by the range pass, except
// `inexact`, which the exact pass sets when a value is off its grid.
struct AccRange {
  int exact;    // the exact path applies
  int narrow;   // ... on the 63-bit grid (every exponent within 10 of the largest)
  int S;        // grid exponent: 62 - Emax (narrow) or 78 - Emax
  int inexact;  // a value fell off the grid
};

// Select state: the three prefixes first (they become the percentiles' bit
// patterns and sit right after the eight sums, so one copy reads both).
struct SelState {
  uint64_t pf[kAccTargets];
  int64_t rk[kAccTargets];  // rank still to find below each prefix
  uint64_t relmax;          // largest rel (its bit pattern)
  int shift;                // bits below the settled prefixes; 0 when done
  int pad;
  // candidate lists after the first digit: target t's samples sit in list
  // slot[t] (targets with the same prefix share one), at cbase[slot] in the
  // candidate buffer, ccnt[t] of them; ccur[] are the append cursors
  int64_t cbase[kAccTargets];
  int64_t ccnt[kAccTargets];
  unsigned long long ccur[kAccTargets];
  int slot[kAccTargets];
  int pad2;
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

// Block maxima of two words, valid in thread 0; `red` holds two words per
// warp.
__device__ __forceinline__ void block_max2(unsigned long long &a, unsigned long long &b, unsigned long long *red) {
#pragma unroll
  for (int d = 16; d; d >>= 1) {
    a = max(a, __shfl_xor_sync(0xffffffffu, a, d));
    b = max(b, __shfl_xor_sync(0xffffffffu, b, d));
  }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) {
    red[2 * wid] = a;
    red[2 * wid + 1] = b;
  }
  __syncthreads();
  if (threadIdx.x == 0)
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) {
      a = max(a, red[2 * w]);
      b = max(b, red[2 * w + 1]);
    }
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

// Largest magnitude (high word of the largest sample y or |T|) and smallest
// exponent over the samples' y and non-zero T, and with them the path: exact
// when the values are finite, n < 2^32 (the integer widths hold any count
// below it) and Emax lies in [kAccEmaxLo, kAccEmaxHi]; narrow (64-bit
// integers) when in addition every exponent is within 10 of Emax.  On the wide
// grid the exact pass checks that every value lies on it.  (A NaN y counts
// here, sending the call to the fp64 path, which leaves it out.)  Block maxima
// go to the partials; the last block folds them.
__global__ void __launch_bounds__(kAccBlock) k_acc_range(const double *__restrict__ y, const double *__restrict__ T,
                                                         int64_t n, AccRange *__restrict__ rg,
                                                         uint64_t *__restrict__ part, unsigned int *ticket) {
  __shared__ unsigned long long red[kAccBlock / 32 * 2];
  unsigned int top = 0u, nmin = 0u;  // nmin: max of 2047 - biased exponent
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i0 = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i0 < n; i0 += 4 * stride) {
    uint2 yv[4], tv[4];  // four elements' loads in flight (a pattern of 0 is not a sample)
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t i = i0 + k * stride;
      yv[k] = i < n ? __ldg(reinterpret_cast<const uint2 *>(y) + i) : make_uint2(0u, 0u);
      tv[k] = i < n ? __ldg(reinterpret_cast<const uint2 *>(T) + i) : make_uint2(0u, 0u);
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const unsigned int yh = yv[k].y, th = tv[k].y & 0x7FFFFFFFu;
      if ((int)yh > 0 || (yh == 0u && yv[k].x != 0u)) {
        top = max(top, max(yh, th));
        nmin = max(nmin, 2047u - (yh >> 20));
        if (th | tv[k].x) nmin = max(nmin, 2047u - (th >> 20));
      }
    }
  }
  unsigned long long a = top, b = nmin;
  block_max2(a, b, red);
  if (threadIdx.x == 0) {
    part[(int64_t)kAccPart * blockIdx.x] = a;
    part[(int64_t)kAccPart * blockIdx.x + 1] = b;
  }
  if (!last_block(ticket)) return;
  a = 0ull;
  b = 0ull;
  for (int k = threadIdx.x; k < (int)gridDim.x; k += kAccBlock) {
    a = max(a, (unsigned long long)__ldcg(part + (int64_t)kAccPart * k));
    b = max(b, (unsigned long long)__ldcg(part + (int64_t)kAccPart * k + 1));
  }
  block_max2(a, b, red);
  if (threadIdx.x == 0) {
    const int E = (int)(a >> 20) - 1023;  // no sample: -1023, and nothing to sum
    const int Emin = 2047 - (int)b - 1023;
    const bool ex = a < 0x7FF00000ull && n < (int64_t)1 << 32 && (b == 0 || (E >= kAccEmaxLo && E <= kAccEmaxHi));
    rg->exact = ex;
    rg->narrow = ex && E - Emin <= 10;
    rg->S = (E - Emin <= 10 ? 62 : kAccGrid) - E;
    rg->inexact = 0;
  }
}

// ---------------------------------------------------------------- exact path

__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// x as a float, truncated to 24 bits (relative error below 2^-23), by bit
// arithmetic on the integer pipe.
__device__ __forceinline__ float acc_u64_to_f32(uint64_t x) {
  const int lz = __clzll((long long)x);
  const uint64_t nx = x << (lz & 63);
  const uint32_t bits = ((uint32_t)(190 - lz) << 23) + (uint32_t)(nx >> 40) - 0x800000u;
  return x ? __uint_as_float(bits) : 0.0f;
}

// floor(e) for 0 <= e < 2^23: adding 2^23 rounded downward leaves it in the
// low mantissa bits.
__device__ __forceinline__ uint32_t acc_floor(float e) {
  return __float_as_uint(__fadd_rd(e, 8388608.0f)) - 0x4B000000u;
}

// q B exactly (q < 2^32, B < 2^64), from two 32 x 32 -> 64-bit products.
__device__ __forceinline__ u128 acc_mul32x64(uint32_t q, uint64_t B) {
  return ((u128)((uint64_t)q * (uint32_t)(B >> 32)) << 32) + (uint64_t)q * (uint32_t)B;
}

// One schoolbook quotient digit: q = floor(R / Bs) given an estimate within
// one of the true digit, R reduced by q Bs.  The remainder after the estimate
// lies in [-Bs, 2 Bs); one conditional add and one conditional subtract settle
// it.  |R| < 2^127 throughout, so the top bit is the sign.
__device__ __forceinline__ uint32_t acc_settle(u128 &R, u128 Bs, u128 qBs, uint32_t q) {
  R -= qBs;
  const bool neg = (uint64_t)(R >> 64) >> 63;
  R += neg ? Bs : (u128)0;
  q -= neg ? 1u : 0u;
  const bool ge = R >= Bs;
  R -= ge ? Bs : (u128)0;
  return q + (ge ? 1u : 0u);
}

// floor(Ma 2^54 / B) for 2^52 <= Ma, B < 2^53 (so the quotient lies in
// [2^53, 2^55)), and whether the remainder is non-zero.  Schoolbook division
// with three digits of 20, 20 and 15 bits: each digit is estimated from a
// single-precision reciprocal of B's top 24 bits and the remainder's top bits
// (relative error below 2^-20.4 all told, so with digits below 2^20 the
// estimate's floor is within one of the true digit) and settled exactly on the
// integer remainder.
__device__ __forceinline__ uint64_t acc_div54(uint64_t Ma, uint64_t B, bool &rem_nz) {
  // B >> 29 lies in [2^23, 2^24): its float is exponent 150 and the low 23 bits
  const float inv = rcp_approx(__uint_as_float((150u << 23) | ((uint32_t)(B >> 29) & 0x7FFFFFu)));
  u128 R = (u128)Ma << 54;
  const u128 B35 = (u128)B << 35, B15 = (u128)B << 15, B0 = (u128)B;
  uint32_t q1 = acc_floor(__fmul_rn(acc_u64_to_f32(Ma >> 10), inv));
  q1 = acc_settle(R, B35, acc_mul32x64(q1, B) << 35, q1);
  uint32_t q2 = acc_floor(__fmul_rn(__fmul_rn(acc_u64_to_f32((uint64_t)(R >> 40)), inv), 0.0625f));
  q2 = acc_settle(R, B15, acc_mul32x64(q2, B) << 15, q2);
  uint32_t q3 = acc_floor(__fmul_rn(__fmul_rn(acc_u64_to_f32((uint64_t)(R >> 20)), inv), 1.0f / 512.0f));
  q3 = acc_settle(R, B0, acc_mul32x64(q3, B), q3);
  rem_nz = R != 0;
  return ((uint64_t)q1 << 35) + ((uint64_t)q2 << 15) + q3;
}

// fl(Ma 2^ka / (My 2^ky)) as a bit pattern, for 2^52 <= Ma, My < 2^53: the
// quotient rounded to nearest (ties to even).  Every quotient here lies in
// [2^-81, 2^81], a normal double.
__device__ __forceinline__ uint64_t acc_quot_bits(uint64_t Ma, int ka, uint64_t My, int ky) {
  bool rem;
  const uint64_t Q = acc_div54(Ma, My, rem);  // quotient = (Q + frac) 2^(ka - ky - 54)
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

// Bit pattern of fl(fl(|D|) / y), where |D| (below 2^80) is |T - y| on the
// grid and y = My 2^ky on the same grid: the difference rounded to 53 bits
// (nearest, ties to even), then the quotient rounded the same way.
__device__ __forceinline__ uint64_t acc_rel_bits(u128 Dm, uint64_t My, int ky) {
  if (Dm == 0) return 0ull;
  const uint64_t dh = (uint64_t)(Dm >> 64), dl = (uint64_t)Dm;
  const int lead = dh ? 127 - __clzll((long long)dh) : 63 - __clzll((long long)dl);
  int ka = lead - 52;
  uint64_t Ma;
  if (ka <= 0) {
    Ma = dl << -ka;
  } else {
    // drop ka (1..27) bits, all in the low word, rounding to nearest even
    Ma = (dl >> ka) | (dh << (64 - ka));
    const uint64_t low = dl & ((1ull << ka) - 1), half = 1ull << (ka - 1);
    Ma += (low > half || (low == half && (Ma & 1ull))) ? 1ull : 0ull;
    const uint64_t carry = Ma >> 53;
    Ma >>= carry;
    ka += (int)carry;
  }
  return acc_quot_bits(Ma, ka, My, ky);
}

// The same for |D| below 2^64.
__device__ __forceinline__ uint64_t acc_rel_bits64(uint64_t d, uint64_t My, int ky) {
  if (d == 0) return 0ull;
  int ka = 63 - __clzll((long long)d) - 52;
  uint64_t Ma;
  if (ka <= 0) {
    Ma = d << -ka;
  } else {
    // drop ka (1..11) bits, rounding to nearest even
    Ma = d >> ka;
    const uint64_t low = d & ((1ull << ka) - 1), half = 1ull << (ka - 1);
    Ma += (low > half || (low == half && (Ma & 1ull))) ? 1ull : 0ull;
    const uint64_t carry = Ma >> 53;
    Ma >>= carry;
    ka += (int)carry;
  }
  return acc_quot_bits(Ma, ka, My, ky);
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

// a += x^2 for x < 2^64 (a: 192 bits).
__device__ __forceinline__ void add_sq64(uint64_t *a, uint64_t x) {
  add192w(a, x * x, __umul64hi(x, x), 0ull);
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

// M 2^k as an integer for k <= 26; `lost` is set when k < 0 drops set bits
// (the value is not on the grid).
__device__ __forceinline__ u128 acc_grid(uint64_t M, int k, bool &lost) {
  const int r = min(-k, 63);
  lost |= k < 0 && (-k > 52 || (M & ((1ull << r) - 1)) != 0ull);
  const uint64_t lo = k >= 0 ? M << k : M >> r;
  const uint64_t hi = k > 0 ? M >> (64 - k) : 0ull;
  return ((u128)hi << 64) | lo;
}

// One sample on the grid 2^-S: the sums and rel's bit pattern.  `lost` is set
// when y or T is not on the grid (the results are then discarded).
__device__ __forceinline__ uint64_t acc_exact_sample(uint64_t yb, uint64_t tb, int S, uint64_t *w, bool &lost) {
  const int bey = (int)(yb >> 52);
  const uint64_t My = (yb & kFracMask) | kHiddenBit;
  const int ky = max(bey, 1) - 1075 + S;  // y = My 2^ky on the grid, ky <= 26
  lost |= bey == 0;                       // subnormal: far below any grid in use
  const u128 Y = acc_grid(My, ky, lost);
  u128 Tm = 0;
  const bool tneg = (tb >> 63) != 0;
  if (tb << 1) {
    const int bet = (int)((tb >> 52) & 0x7FF);
    Tm = acc_grid((tb & kFracMask) | (bet ? kHiddenBit : 0ull), max(bet, 1) - 1075 + S, lost);
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

// One sample on the 63-bit grid 2^-S (every exponent within 10 of the
// largest, so each value is an integer below 2^63 there): the sums and rel's
// bit pattern.
__device__ __forceinline__ uint64_t acc_exact_sample64(uint64_t yb, uint64_t tb, int S, uint64_t *w) {
  const uint64_t My = (yb & kFracMask) | kHiddenBit;
  const int ky = (int)(yb >> 52) - 1075 + S;  // 0..10
  const uint64_t Y = My << ky;
  uint64_t Tm = 0ull;
  const bool tneg = (tb >> 63) != 0;
  if (tb << 1) Tm = ((tb & kFracMask) | kHiddenBit) << ((int)((tb >> 52) & 0x7FF) - 1075 + S);
  w[0] += 1;
  add128w(w + 1, Y);
  add128w(w + 3, tneg ? (u128)0 - Tm : (u128)Tm);
  const uint64_t Dm = tneg ? Y + Tm : (Y >= Tm ? Y - Tm : Tm - Y);
  add_sq64(w + 5, Y);
  add_sq64(w + 8, Tm);
  add_sq64(w + 11, Dm);
  return acc_rel_bits64(Dm, My, ky);
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

// The signed 256-bit two's-complement integer w, times 2^e2, as the nearest
// double (ties to even), by integer operations only; `ok` is cleared when the
// result would leave the normal range (the caller then takes a slower route).
__device__ __forceinline__ double acc_i256_to_double(const uint64_t *wi, int e2, bool &ok) {
  uint64_t w0 = wi[0], w1 = wi[1], w2 = wi[2], w3 = wi[3];
  const bool neg = (w3 >> 63) != 0;
  if (neg) {
    w0 = ~w0;
    w1 = ~w1;
    w2 = ~w2;
    w3 = ~w3;
    u128 s = (u128)w0 + 1;
    w0 = (uint64_t)s;
    s = (u128)w1 + (uint64_t)(s >> 64);
    w1 = (uint64_t)s;
    s = (u128)w2 + (uint64_t)(s >> 64);
    w2 = (uint64_t)s;
    w3 += (uint64_t)(s >> 64);
  }
  const int t = w3 ? 3 : w2 ? 2 : w1 ? 1 : 0;
  const uint64_t a = t == 3 ? w3 : t == 2 ? w2 : t == 1 ? w1 : w0;
  if (a == 0) return 0.0;
  const uint64_t b = t == 3 ? w2 : t == 2 ? w1 : t == 1 ? w0 : 0ull;
  const bool rest = (t == 3 ? (w1 | w0) : t == 2 ? w0 : 0ull) != 0ull;
  const int lz = __clzll((long long)a);
  const uint64_t top = lz ? (a << lz) | (b >> (64 - lz)) : a;  // leading one at bit 63
  const bool below = (lz ? (b << lz) : b) != 0ull || rest;
  uint64_t mant = top >> 11;
  const uint64_t rb = (top >> 10) & 1ull;
  const bool st = (top & 0x3FFull) != 0ull || below;
  mant += rb & ((st ? 1ull : 0ull) | (mant & 1ull));
  int ex = 64 * t + 63 - lz + e2;  // exponent of the leading bit
  if (mant >> 53) {
    mant >>= 1;
    ++ex;
  }
  if (ex < -1022 || ex > 1023) {
    ok = false;
    return 0.0;
  }
  return __longlong_as_double((long long)(((uint64_t)neg << 63) | ((uint64_t)(ex + 1023) << 52) | (mant & kFracMask)));
}

// Select state for a new call: the prefix every sample shares (the common
// leading bits of the smallest and largest rel, lo and hi) and the target
// ranks ceil(q m / 100), q = 50, 90, 99.
__device__ __forceinline__ void acc_publish_select(uint64_t hi, uint64_t lo, SelState *sel, int64_t m) {
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

// Largest rel and largest ~rel (so zero is the identity of both).
__device__ __forceinline__ void acc_note_rel(uint64_t rb, unsigned long long &rmax, unsigned long long &rnmax) {
  rmax = max(rmax, (unsigned long long)rb);
  rnmax = max(rnmax, (unsigned long long)~rb);
}

template <bool kNarrow>
__device__ __forceinline__ void acc_exact_loop(const double *__restrict__ y, const double *__restrict__ T, int64_t n,
                                               int S, uint64_t *__restrict__ relbits, uint64_t *w,
                                               unsigned long long &rmax, unsigned long long &rnmax, bool &lost) {
  const int64_t stride = (int64_t)gridDim.x * kAccBlock;
  for (int64_t i0 = blockIdx.x * (int64_t)kAccBlock + threadIdx.x; i0 < n; i0 += 2 * stride) {
    uint64_t yb[2], tb[2];  // two elements' loads in flight (a pattern of 0 is not a sample)
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int64_t i = i0 + k * stride;
      yb[k] = i < n ? (uint64_t)__double_as_longlong(__ldg(y + i)) : 0ull;
      tb[k] = i < n ? (uint64_t)__double_as_longlong(__ldg(T + i)) : 0ull;
    }
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      const int64_t i = i0 + k * stride;
      uint64_t rb = ~0ull;  // not a sample
      if (acc_is_sample(yb[k])) {
        rb = kNarrow ? acc_exact_sample64(yb[k], tb[k], S, w) : acc_exact_sample(yb[k], tb[k], S, w, lost);
        acc_note_rel(rb, rmax, rnmax);
      }
      if (i < n) relbits[i] = rb;
    }
  }
}

// Exact path: the sums and every rel in one pass over y and T; the last block
// folds the block partials and writes sums[0] = m and, scaled by m 2^(2S),
// sums[3..6] = sxx, syy, sxy, ssr.  Returns at once when the range pass chose
// the fp64 path; flags rg->inexact (and the fp64 path then redoes the call)
// when a value is not on the grid.
__global__ void __launch_bounds__(kAccBlock) k_acc_exact(const double *__restrict__ y, const double *__restrict__ T,
                                                         int64_t n, AccRange *__restrict__ rg,
                                                         uint64_t *__restrict__ relbits, uint64_t *__restrict__ part,
                                                         double *__restrict__ sums, SelState *__restrict__ sel,
                                                         unsigned int *ticket) {
  __shared__ uint64_t red[kAccBlock / 32 * kAccWords];
  __shared__ unsigned long long red2[kAccBlock / 32 * 2];
  if (!rg->exact) return;
  const int S = rg->S;
  uint64_t w[kAccWords];
#pragma unroll
  for (int j = 0; j < kAccWords; ++j) w[j] = 0ull;
  unsigned long long rmax = 0ull, rnmax = 0ull;
  bool lost = false;
  if (rg->narrow)
    acc_exact_loop<true>(y, T, n, S, relbits, w, rmax, rnmax, lost);
  else
    acc_exact_loop<false>(y, T, n, S, relbits, w, rmax, rnmax, lost);
  if (__syncthreads_or(lost) && threadIdx.x == 0) atomicOr(&rg->inexact, 1);
  block_max2(rmax, rnmax, red2);
  acc_block_combine(w, red);
  if (threadIdx.x == 0) {
    uint64_t *p = part + (int64_t)blockIdx.x * kAccPart;
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) p[j] = w[j];
    p[kAccWords] = rmax;
    p[kAccWords + 1] = rnmax;
  }
  if (!last_block(ticket)) return;
#pragma unroll
  for (int j = 0; j < kAccWords; ++j) w[j] = 0ull;
  rmax = rnmax = 0ull;
  for (int b = threadIdx.x; b < (int)gridDim.x; b += kAccBlock) {
    const uint64_t *p = part + (int64_t)b * kAccPart;
    uint64_t o[kAccWords];
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) o[j] = __ldcg(p + j);
    acc_combine(w, o);
    rmax = max(rmax, (unsigned long long)__ldcg(p + kAccWords));
    rnmax = max(rnmax, (unsigned long long)__ldcg(p + kAccWords + 1));
  }
  block_max2(rmax, rnmax, red2);
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
  bool ok = true;  // every value here is below 2^227 in magnitude
  sums[0] = (double)m;
  sums[3] = acc_i256_to_double(sxx, 0, ok);
  sums[4] = acc_i256_to_double(syy, 0, ok);
  sums[5] = acc_i256_to_double(sxy, -1, ok);
  sums[6] = acc_i256_to_double(ssr, 0, ok);
  acc_publish_select(rmax, ~(uint64_t)rnmax, sel, (int64_t)m);
}

// ---------------------------------------------------------------- fp64 path

// Pass 1: per-block count, sum y, sum T over the samples; rel's bit patterns
// stored (all ones for a batch that is not a sample, which the select never
// counts).  The last block folds the partials into sums[0..2] and sets up the
// select.  Returns at once when the exact path did the call.
__global__ void __launch_bounds__(kAccBlock) k_acc_sums(const double *__restrict__ y, const double *__restrict__ T,
                                                        int64_t n, const AccRange *__restrict__ rg,
                                                        uint64_t *__restrict__ relbits, double *__restrict__ part,
                                                        double *__restrict__ sums, SelState *__restrict__ sel,
                                                        unsigned int *ticket) {
  __shared__ double red[kAccBlock / 32];
  __shared__ unsigned long long red2[kAccBlock / 32 * 2];
  if (rg->exact && !rg->inexact) return;
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
  block_max2(rmax, rnmax, red2);
  const double a = block_sum_fixed(c, red), b = block_sum_fixed(sy, red), d = block_sum_fixed(st, red);
  if (threadIdx.x == 0) {
    double *p = part + (int64_t)kAccPart * blockIdx.x;
    p[0] = a;
    p[1] = b;
    p[2] = d;
    p[3] = __longlong_as_double((long long)rmax);  // bit patterns, folded as integers
    p[4] = __longlong_as_double((long long)rnmax);
  }
  if (!last_block(ticket)) return;
  fold_partials(part, gridDim.x, 3, red, sums);
  rmax = rnmax = 0ull;
  for (int k = threadIdx.x; k < (int)gridDim.x; k += kAccBlock) {
    const double *p = part + (int64_t)kAccPart * k;
    rmax = max(rmax, (unsigned long long)__double_as_longlong(__ldcg(p + 3)));
    rnmax = max(rnmax, (unsigned long long)__double_as_longlong(__ldcg(p + 4)));
  }
  block_max2(rmax, rnmax, red2);
  if (threadIdx.x == 0) acc_publish_select(rmax, ~(uint64_t)rnmax, sel, (int64_t)sums[0]);
}

// Pass 2: centred moments with the means from pass 1 (sums = {count, sum y,
// sum T}); the last block folds them into sums[3..6] = sxx, syy, sxy, ssr.
__global__ void __launch_bounds__(kAccBlock) k_acc_moments(const double *__restrict__ y, const double *__restrict__ T,
                                                           int64_t n, const AccRange *__restrict__ rg,
                                                           double *__restrict__ sums, double *__restrict__ part,
                                                           unsigned int *ticket) {
  __shared__ double red[kAccBlock / 32];
  if (rg->exact && !rg->inexact) return;
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


// One warp: the bin of a kSelBins-bin histogram that holds rank r (1-based),
// the count below that bin and the bin's own count, valid in every lane.  Lane
// l sums bins [64 l, 64 l + 64), a warp scan finds the lane whose range holds
// r, then the same over that lane's bins two at a time.  kGlobal: the
// histogram is in global memory, written by other blocks' atomics.
template <bool kGlobal>
__device__ __forceinline__ void acc_scan_pick(const unsigned int *h, int64_t r, int &bin, int64_t &below,
                                              int64_t &cnt) {
  static_assert(kSelBins == 64 * 32, "64 bins per lane");
  const int lane = threadIdx.x & 31;
  int64_t s = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint4 *p = reinterpret_cast<const uint4 *>(h + 64 * lane + 4 * j);
    const uint4 q = kGlobal ? __ldcg(p) : *p;
    s += (int64_t)q.x + q.y + q.z + q.w;
  }
  int64_t inc = s;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int64_t o = __shfl_up_sync(0xffffffffu, inc, d);
    if (lane >= d) inc += o;
  }
  unsigned ball = __ballot_sync(0xffffffffu, inc >= r);
  const int L = ball ? __ffs(ball) - 1 : 31;
  const int64_t bl = __shfl_sync(0xffffffffu, inc - s, L);
  const uint2 *p2 = reinterpret_cast<const uint2 *>(h + 64 * L + 2 * lane);
  const uint2 pr = kGlobal ? __ldcg(p2) : *p2;
  const int64_t ps = (int64_t)pr.x + pr.y;
  int64_t inc2 = ps;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int64_t o = __shfl_up_sync(0xffffffffu, inc2, d);
    if (lane >= d) inc2 += o;
  }
  ball = __ballot_sync(0xffffffffu, bl + inc2 >= r);
  const int L2 = ball ? __ffs(ball) - 1 : 31;
  const int64_t b0 = bl + inc2 - ps;
  const bool first = b0 + pr.x >= r;
  bin = __shfl_sync(0xffffffffu, 64 * L + 2 * lane + (first ? 0 : 1), L2);
  below = __shfl_sync(0xffffffffu, first ? b0 : b0 + (int64_t)pr.x, L2);
  cnt = __shfl_sync(0xffffffffu, (int64_t)(first ? pr.x : pr.y), L2);
}

// Select, first digit: every sample adds one to the histogram of its first
// digit below the shared prefix (all samples share it, so no compare), and
// its rel to the fixed-point sum.  The last block writes sums[7] (the largest
// rel itself when that is inf or NaN, which is what an exact sum gives then),
// picks each target's digit, and lays out the candidate lists: targets in the
// same bin share one.  With no digit left (every rel equal) the prefixes are
// already the answers.
__global__ void __launch_bounds__(kSelBlock) k_acc_sel0(const uint64_t *__restrict__ relbits, int64_t n,
                                                        SelState *__restrict__ sel, unsigned int *__restrict__ hist,
                                                        uint64_t *__restrict__ part, double *__restrict__ sums,
                                                        unsigned int *ticket) {
  __shared__ unsigned int h[kSelBins];
  __shared__ uint64_t red[kSelBlock / 32 * 3];
  const int shift = sel->shift;
  const uint64_t relmax = sel->relmax;
  const bool digit = shift > 0;
  const bool rsum = relmax < 0x7FF0000000000000ull;
  const int w = min(kSelBits, shift), lo = shift - w;
  const uint64_t dmask = (1ull << w) - 1;
  for (int i = threadIdx.x; i < kSelBins; i += kSelBlock) h[i] = 0u;
  __syncthreads();
  const int bemax = max((int)(relmax >> 52), 1);
  uint64_t acc[3] = {0, 0, 0};  // sum of rel on its grid, 192 bits
  auto visit = [&](uint64_t v) {
    if (v == ~0ull) return;  // not a sample
    if (digit) atomicAdd(&h[(int)((v >> lo) & dmask)], 1u);
    if (rsum) {
      const u128 x = acc_rel_fixed(v, bemax);
      add192w(acc, (uint64_t)x, (uint64_t)(x >> 64), 0);
    }
  };
  // eight consecutive patterns per thread (four 16-byte loads in flight), then the tail
  const int64_t n8 = n >> 3;
  const int64_t g = blockIdx.x * (int64_t)kSelBlock + threadIdx.x, stride = (int64_t)gridDim.x * kSelBlock;
  const ulonglong2 *r2 = reinterpret_cast<const ulonglong2 *>(relbits);
  for (int64_t c = g; c < n8; c += stride) {
    ulonglong2 q[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) q[k] = __ldcg(r2 + 4 * c + k);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      visit(q[k].x);
      visit(q[k].y);
    }
  }
  if (g < n - 8 * n8) visit(__ldcg(relbits + 8 * n8 + g));
  __syncthreads();
  if (digit)
    for (int i = threadIdx.x; i < kSelBins; i += kSelBlock) {
      const unsigned int c = h[i];
      if (c) atomicAdd(hist + i, c);
    }
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int d = 16; d; d >>= 1) {
    const uint64_t o0 = __shfl_xor_sync(0xffffffffu, acc[0], d), o1 = __shfl_xor_sync(0xffffffffu, acc[1], d),
                   o2 = __shfl_xor_sync(0xffffffffu, acc[2], d);
    add192w(acc, o0, o1, o2);
  }
  if (lane == 0) {
    red[3 * wid] = acc[0];
    red[3 * wid + 1] = acc[1];
    red[3 * wid + 2] = acc[2];
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int v = 1; v < kSelBlock / 32; ++v) add192w(acc, red[3 * v], red[3 * v + 1], red[3 * v + 2]);
    uint64_t *p = part + (int64_t)kAccPart * blockIdx.x;
    p[0] = acc[0];
    p[1] = acc[1];
    p[2] = acc[2];
  }
  if (!last_block(ticket)) return;
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
    bool ok = true;
    double sr = rsum ? acc_i256_to_double(wv, bemax - 1123, ok) : __longlong_as_double((long long)relmax);
    if (!ok) sr = ldexp(int256_to_dd(wv, 0).hi, bemax - 1123);  // sums below 2^-1022 or above 2^1023
    sums[7] = sr;
  }
  if (!digit) return;
  __shared__ uint64_t npf[kAccTargets];
  __shared__ int64_t nrk[kAccTargets];
  __syncthreads();
  for (int i = threadIdx.x; i < kSelBins; i += kSelBlock) h[i] = __ldcg(hist + i);  // the grid's histogram
  __syncthreads();
  if (wid < kAccTargets) {
    int bin;
    int64_t below, cnt;
    const int64_t r = sel->rk[wid];
    acc_scan_pick<false>(h, r, bin, below, cnt);
    if (lane == 0) {
      npf[wid] = (sel->pf[wid] << w) | (uint64_t)bin;
      nrk[wid] = r - below;
    }
  }
  __syncthreads();
  if (threadIdx.x < kAccTargets) {
    sel->pf[threadIdx.x] = npf[threadIdx.x];
    sel->rk[threadIdx.x] = nrk[threadIdx.x];
  }
  if (threadIdx.x == 0) sel->shift = lo;
  for (int i = threadIdx.x; i < kSelBins; i += kSelBlock) hist[i] = 0u;
}

// Select, second digit: a sample whose bits above `shift` equal a target's
// prefix adds one, in global memory, to that prefix's histogram at its next
// digit (few samples do: those in a first-digit bin that holds a target).
// Prefixes of one length are equal or disjoint, so a sample counts at most
// once; targets with the same prefix share a histogram.  The last block picks
// each target's digit and lays out the candidate lists for the gather:
// targets whose bins coincide share one, of that bin's count.
__global__ void __launch_bounds__(kSelBlock) k_acc_selB(const uint64_t *__restrict__ relbits, int64_t n,
                                                        SelState *__restrict__ sel, unsigned int *__restrict__ hist,
                                                        unsigned int *ticket) {
  __shared__ unsigned int h[kAccTargets * kSelBins];
  __shared__ uint64_t npf[kAccTargets];
  __shared__ int64_t nrk[kAccTargets], ncnt[kAccTargets];
  const int shift = sel->shift;
  if (shift <= 0) return;
  const uint64_t pf0 = sel->pf[0], pf1 = sel->pf[1], pf2 = sel->pf[2];
  const int w = min(kSelBits, shift), lo = shift - w;
  const uint64_t dmask = (1ull << w) - 1;
  auto visit = [&](uint64_t v) {
    if (v == ~0ull) return;  // not a sample
    const uint64_t key = v >> shift;
    const int s = key == pf0 ? 0 : key == pf1 ? 1 : key == pf2 ? 2 : -1;
    if (s >= 0) atomicAdd(hist + s * kSelBins + (int)((v >> lo) & dmask), 1u);
  };
  const int64_t n8 = n >> 3;
  const int64_t g = blockIdx.x * (int64_t)kSelBlock + threadIdx.x, stride = (int64_t)gridDim.x * kSelBlock;
  const ulonglong2 *r2 = reinterpret_cast<const ulonglong2 *>(relbits);
  for (int64_t c = g; c < n8; c += stride) {
    ulonglong2 q[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) q[k] = __ldcg(r2 + 4 * c + k);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      visit(q[k].x);
      visit(q[k].y);
    }
  }
  if (g < n - 8 * n8) visit(__ldcg(relbits + 8 * n8 + g));
  if (!last_block(ticket)) return;
  for (int i = threadIdx.x; i < kAccTargets * kSelBins; i += kSelBlock) h[i] = __ldcg(hist + i);
  __syncthreads();
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (wid < kAccTargets) {
    const uint64_t pf = wid == 0 ? pf0 : wid == 1 ? pf1 : pf2;
    const int slot = pf == pf0 ? 0 : pf == pf1 ? 1 : 2;
    const int64_t r = sel->rk[wid];
    int bin;
    int64_t below, cnt;
    acc_scan_pick<false>(h + slot * kSelBins, r, bin, below, cnt);
    if (lane == 0) {
      npf[wid] = (pf << w) | (uint64_t)bin;
      nrk[wid] = r - below;
      ncnt[wid] = cnt;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // candidate lists: targets whose bins coincide share one, of that bin's count
    int sl[kAccTargets];
    int64_t base = 0;
    for (int t = 0; t < kAccTargets; ++t) {
      sl[t] = t;
      for (int u = t - 1; u >= 0; --u)
        if (npf[u] == npf[t]) sl[t] = sl[u];
      sel->pf[t] = npf[t];
      sel->rk[t] = nrk[t];
      sel->ccnt[t] = ncnt[t];
      sel->slot[t] = sl[t];
      if (sl[t] == t) {
        sel->cbase[t] = base;
        base += ncnt[t];
      }
    }
    sel->shift = lo;
  }
  for (int i = threadIdx.x; i < kAccTargets * kSelBins; i += kSelBlock) hist[i] = 0u;
}

// Select, gather: each sample whose bits above `shift` equal a target's
// prefix is appended to that prefix's candidate list (a sample joins at most
// one list, and each list's length is its bin's count).  A block counts its
// samples per list, reserves its ranges with one atomic per list, and writes
// them; the order within a list does not matter.
__global__ void __launch_bounds__(kSelBlock) k_acc_sel1(const uint64_t *__restrict__ relbits, int64_t n,
                                                        SelState *__restrict__ sel, uint64_t *__restrict__ cand) {
  __shared__ int wofs[kSelBlock / 32][kAccTargets];
  __shared__ unsigned long long bbase[kAccTargets];
  const int shift = sel->shift;
  if (shift <= 0) return;
  const uint64_t pf0 = sel->pf[0], pf1 = sel->pf[1], pf2 = sel->pf[2];
  const int64_t base0 = sel->cbase[0], base1 = sel->cbase[1], base2 = sel->cbase[2];
  const int64_t cnt0 = sel->ccnt[0], cnt1 = sel->ccnt[1], cnt2 = sel->ccnt[2];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const int64_t nc = (n + 7) >> 3;  // chunks of eight patterns, the last one padded
  for (int64_t cb = blockIdx.x * (int64_t)kSelBlock; cb < nc; cb += (int64_t)gridDim.x * kSelBlock) {
    const int64_t c = cb + threadIdx.x;
    uint64_t v[8];
    const bool full = 8 * c + 8 <= n;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      ulonglong2 q;
      if (full) {
        q = __ldcg(reinterpret_cast<const ulonglong2 *>(relbits) + 4 * c + k);
      } else {
        const int64_t i = 8 * c + 2 * k;
        q.x = i < n ? __ldcg(relbits + i) : ~0ull;
        q.y = i + 1 < n ? __ldcg(relbits + i + 1) : ~0ull;
      }
      v[2 * k] = q.x;
      v[2 * k + 1] = q.y;
    }
    uint32_t sl = 0;  // two bits per pattern: its list, 3 for none
    int own[kAccTargets] = {0, 0, 0};
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      uint32_t s = 3u;
      if (v[k] != ~0ull) {
        const uint64_t key = v[k] >> shift;
        s = key == pf0 ? 0u : key == pf1 ? 1u : key == pf2 ? 2u : 3u;
      }
      sl |= s << (2 * k);
#pragma unroll
      for (int j = 0; j < kAccTargets; ++j) own[j] += s == (uint32_t)j ? 1 : 0;
    }
    int before[kAccTargets];  // this thread's offset within its warp, per list
#pragma unroll
    for (int j = 0; j < kAccTargets; ++j) {
      int inc = own[j];
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int o = __shfl_up_sync(0xffffffffu, inc, d);
        if (lane >= d) inc += o;
      }
      before[j] = inc - own[j];
      if (lane == 31) wofs[wid][j] = inc;
    }
    __syncthreads();
    if (threadIdx.x < kAccTargets) {
      const int j = threadIdx.x;
      int run = 0;
      for (int u = 0; u < kSelBlock / 32; ++u) {
        const int t = wofs[u][j];
        wofs[u][j] = run;
        run += t;
      }
      bbase[j] = run ? atomicAdd(&sel->ccur[j], (unsigned long long)run) : 0ull;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 8; ++k)
#pragma unroll
      for (int j = 0; j < kAccTargets; ++j)
        if (((sl >> (2 * k)) & 3u) == (uint32_t)j) {
          const int64_t pos = (int64_t)bbase[j] + wofs[wid][j] + before[j];
          before[j] += 1;
          const int64_t cj = j == 0 ? cnt0 : j == 1 ? cnt1 : cnt2, bj = j == 0 ? base0 : j == 1 ? base1 : base2;
          if (pos < cj) cand[bj + pos] = v[k];
        }
    __syncthreads();
  }
}

// Select, finish: one block per target finds its rank in its candidate list,
// writes the percentile's bit pattern and resets its append cursor.  A list
// of at most one pattern per thread is ranked directly; a longer one is
// settled digit by digit (from the common prefix of its smallest and largest
// pattern on, one shared-memory histogram per digit), from shared memory when
// it fits there (kSelSmemList patterns), else from global memory.
__global__ void __launch_bounds__(kSelFinish) k_acc_sel2(const uint64_t *__restrict__ cand,
                                                         SelState *__restrict__ sel) {
  extern __shared__ uint64_t lst[];  // kSelSmemList patterns (dynamic)
  __shared__ unsigned int h[kSelBins];
  __shared__ unsigned long long mm[2];
  __shared__ int64_t pick[2];
  const int t = blockIdx.x;
  if (sel->shift <= 0) return;
  const uint64_t *list = cand + sel->cbase[sel->slot[t]];
  const int64_t c = sel->ccnt[t];
  int64_t r = sel->rk[t];
  if (c <= 0) return;  // cannot happen: a bin that holds a rank is not empty
  if (c <= kSelFinish) {
    // a short list: the candidate with fewer than r smaller ones and at least
    // r not larger is the answer (every thread that finds it holds the same value)
    if (threadIdx.x < c) lst[threadIdx.x] = __ldcg(list + threadIdx.x);
    __syncthreads();
    if (threadIdx.x < c) {
      const uint64_t v = lst[threadIdx.x];
      int64_t less = 0, leq = 0;
      for (int j = 0; j < (int)c; ++j) {
        const uint64_t u = lst[j];
        less += u < v ? 1 : 0;
        leq += u <= v ? 1 : 0;
      }
      if (less < r && r <= leq) sel->pf[t] = v;
    }
    if (threadIdx.x == 0) sel->ccur[t] = 0ull;
    return;
  }
  const bool inshared = c <= kSelSmemList;
  if (threadIdx.x == 0) {
    mm[0] = 0ull;
    mm[1] = 0ull;
  }
  unsigned long long mx = 0ull, nmn = 0ull;
  for (int64_t i = threadIdx.x; i < c; i += kSelFinish) {
    const unsigned long long v = __ldcg(list + i);
    if (inshared) lst[i] = v;
    mx = max(mx, v);
    nmn = max(nmn, ~v);
  }
#pragma unroll
  for (int d = 16; d; d >>= 1) {
    mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, d));
    nmn = max(nmn, __shfl_xor_sync(0xffffffffu, nmn, d));
  }
  __syncthreads();
  if ((threadIdx.x & 31) == 0) {
    atomicMax(&mm[0], mx);
    atomicMax(&mm[1], nmn);
  }
  __syncthreads();
  const uint64_t hi = mm[0], lo0 = ~(uint64_t)mm[1];
  int cur = hi == lo0 ? 0 : 64 - __clzll((long long)(hi ^ lo0));
  uint64_t prefix = cur == 0 ? hi : hi >> cur;
  while (cur > 0) {
    const int w = min(kSelBits, cur), lo = cur - w;
    const uint64_t dmask = (1ull << w) - 1;
    for (int i = threadIdx.x; i < kSelBins; i += kSelFinish) h[i] = 0u;
    __syncthreads();
    for (int64_t i = threadIdx.x; i < c; i += kSelFinish) {
      const uint64_t v = inshared ? lst[i] : __ldcg(list + i);
      if ((v >> cur) == prefix) atomicAdd(&h[(int)((v >> lo) & dmask)], 1u);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      int bin;
      int64_t below, cnt;
      acc_scan_pick<false>(h, r, bin, below, cnt);
      if (threadIdx.x == 0) {
        pick[0] = bin;
        pick[1] = below;
      }
    }
    __syncthreads();
    r -= pick[1];
    prefix = (prefix << w) | (uint64_t)pick[0];
    cur = lo;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    sel->pf[t] = prefix;
    sel->ccur[t] = 0ull;
  }
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
