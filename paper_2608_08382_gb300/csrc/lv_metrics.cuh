// Accuracy of predicted batch latencies against measured ones (Section 3.2,
// Tables 1-2: R^2 and percentiles of the relative error), over the samples,
// the batches with y > 0 (m of them):
//   r2_ssr  = 1 - sum (y - T)^2 / sum (y - mean y)^2
//   r2_corr = (sum (y - mean y)(T - mean T))^2 / (sum (y - mean y)^2 sum (T - mean T)^2)
//   rel_b   = |T_b - y_b| / y_b (difference and quotient each rounded to
//             double, as fp64 arithmetic gives them), its mean and its
//             nearest-rank p50, p90, p99 (the ceil(q m / 100)-th smallest).
//
// One cooperative kernel computes all of it.  Its phases are separated by a
// grid-wide barrier; after one, every block derives what it needs from small
// shared results itself (in the same order, so all blocks agree).  Block b
// owns one contiguous range of the batches.
//   range   the largest and smallest binary exponents Emax, Emin among the
//           samples' y and non-zero T.  GB300 issues fp64 at 1/64 of the fp32
//           rate, so when Emax is finite and moderate the sums are formed
//           exactly on the integer pipes: on the grid 2^(Emax - 62) in 64-bit
//           integers when Emax - Emin <= 10 (every value then lies on it), else
//           on 2^(Emax - 78) in 128-bit integers.
//   exact   per sample the integers Y = y 2^S and T 2^S and D = Y - T; the
//           exact sums of Y, T, Y^2, T^2 and D^2, from which
//             m sxx = m sum Y^2 - (sum Y)^2,   m syy = m sum T^2 - (sum T)^2,
//             2 m sxy = m (sum Y^2 + sum T^2 - sum D^2) - 2 sum Y sum T,
//             m ssr = m sum D^2
//           follow exactly (all on the grid 2^(-2S), which both R^2 cancel);
//           rel by exact integer division; the mean of rel as an fp64 sum in
//           a fixed order.  A value off the wide grid sends the call to the
//           fp64 phases.
//   fp64    otherwise (a non-finite sample value, extreme magnitudes, a value
//           off the grid): rel, means, then centred moments, each in a fixed
//           order.
//   select  the percentiles, exact: rel is a non-negative double, so its bit
//           pattern orders like its value, and a most-significant-digit radix
//           select finds the bit pattern of the element of each target rank.
//           The pass that forms rel also histograms its first digit (exponent
//           and top mantissa bits) and sorts each block's samples by it, so a
//           target's first-digit bin is one short segment per block (typically
//           well under 1% of the samples in all).  The next phase histograms
//           the next 11 bits of those segments, keeping each second-digit bin's
//           first samples in a bucket; the block of each target then picks its
//           second digit and ranks the bin's samples (from the bucket, or the
//           blocks' segments when the bin outgrew it).
#pragma once

#include <cstdint>

#include "lv_fit.cuh"

namespace lv {

typedef unsigned __int128 u128;

constexpr int kAccBlock = 256;
constexpr int kAccTargets = 3;  // p50, p90, p99
constexpr int kAccWords = 14;   // the exact sums of one block
constexpr int kSelBits = 11;    // radix digit
constexpr int kSelBins = 1 << kSelBits;
constexpr int kAccStage = 8192;  // a block's rel values kept in shared memory when its range fits
constexpr int kAccBucket = 64;   // samples kept per second-digit bin
constexpr int kAccGrid = 78;  // wide grid: S = kAccGrid - Emax puts every |v 2^S| below 2^79
// Range of Emax for the exact path: within it the definition's own fp64
// arithmetic (squared deviations, their products in r2_corr) neither overflows
// nor underflows for values on the grid, so the exact results are what fp64
// evaluation approximates.
constexpr int kAccEmaxLo = -160, kAccEmaxHi = 224;
constexpr uint64_t kFracMask = (1ull << 52) - 1, kHiddenBit = 1ull << 52;

// One block's partial, kAccPartW words: sample count, rel sum (fp64), the
// range maxima, the exact sums, the fp64 sums (count, sum y, sum T) and the
// fp64 centred moments.
constexpr int kAccPartW = 32;
constexpr int kPC = 0, kPQ = 2, kPR = 4, kPX = 8, kPS = 22, kPM = 25;
static_assert(kPX + kAccWords <= kPS && kPS + 3 <= kPM && kPM + 4 <= kAccPartW, "partial layout");

// Device arguments of one call.  `res` receives the eight sums (m, -, -,
// sxx, syy, sxy, ssr, sum rel), the three percentiles' bit patterns and an
// error word, in host memory the device writes directly.
struct AccArgs {
  const double *y, *T;
  int64_t n;
  uint64_t *relbits;          // n rel bit patterns (all ones: not a sample)
  uint64_t *cand;             // each block's samples sorted by first digit within its range, n patterns
  uint64_t *segs;             // per block and first-digit slot: offset and length of its segment
  uint64_t *bucket;           // kAccTargets * kSelBins buckets of kAccBucket patterns
  uint64_t *part;             // kAccPartW words per block
  double *res;                // results (host memory, mapped): 8 sums, 3 patterns, error word
  int *err;                   // the barrier's error word (device memory)
  int *lost;                  // set when a value is off the wide grid (device memory)
  unsigned int *hist1;        // 2 * kSelBins: first digit, exact pass then fp64 pass
  unsigned int *hist2;        // kAccTargets * kSelBins: the second digit
  unsigned int *bar;          // grid barrier: arrivals, generation (zero between calls)
};

// y > 0 on the bit pattern: sign clear, not zero, not NaN (+inf counts).
__device__ __forceinline__ bool acc_is_sample(uint64_t b) {
  return (int64_t)b > 0 && b <= 0x7FF0000000000000ull;
}

// Grid-wide barrier of a cooperative launch (every block resident).  Thread 0
// of each block arrives on bar[0] with release ordering (the block's earlier
// writes become visible with it); the last arrival resets the count and
// advances the generation bar[1]; the others wait, with acquire ordering, for
// the generation to move, for at most a few seconds, after which they set
// the error word and go on.  Returns false once the error word is set (every
// block then leaves).
__device__ __forceinline__ bool grid_barrier(unsigned int *bar, int *err) {
  __shared__ int ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned int g, old;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(g) : "l"(bar + 1) : "memory");
    asm volatile("atom.add.acq_rel.gpu.global.u32 %0, [%1], 1;" : "=r"(old) : "l"(bar) : "memory");
    if (old == gridDim.x - 1) {
      asm volatile("st.relaxed.gpu.global.u32 [%0], 0;" ::"l"(bar) : "memory");
      asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(bar + 1) : "memory");
    } else {
      unsigned int now;
      for (long long k = 0;; ++k) {
        asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(now) : "l"(bar + 1) : "memory");
        if (now != g) break;
        if (k > (1ll << 24)) {
          atomicExch(err, 1);
          break;
        }
        __nanosleep(20);
      }
    }
    ok = *(volatile int *)err == 0;
  }
  __syncthreads();
  return ok;
}

// A block leaving after a barrier timed out: mark the call failed.
__device__ __forceinline__ void acc_left(const AccArgs &a) {
  if (threadIdx.x == 0) *reinterpret_cast<volatile int *>(a.res + 11) = 1;
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

// ---------------------------------------------------------------- exact path

__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// floor(Ma 2^54 / B) for 2^52 <= Ma, B < 2^53 (so the quotient lies in
// [2^53, 2^55)), and whether the remainder is non-zero.  Through a 64-bit
// reciprocal V ~ 2^116 / B: a single-precision reciprocal of B's top 24 bits
// (relative error about 2^-21) refined by two Newton-Raphson steps
// V += V (2^116 - B V) / 2^116, each squaring the error, to within a few units
// of 2^116 / B; then the quotient estimate Ma V / 2^62, which lies at most one
// below the true quotient, settled on the exact remainder Ma 2^54 - Q B
// (below 2^64 in magnitude, so formed modulo 2^64).  The products run on the
// multiply-add pipe.
__device__ __forceinline__ uint64_t acc_div54(uint64_t Ma, uint64_t B, bool &rem_nz) {
  // B >> 29 lies in [2^23, 2^24): its float is exponent 150 and the low 23 bits
  const uint32_t fb = __float_as_uint(rcp_approx(__uint_as_float((150u << 23) | ((uint32_t)(B >> 29) & 0x7FFFFFu))));
  const int sh = (int)(fb >> 23) - 63;  // the reciprocal lies in (2^-24, 2^-23]: 40 or 41
  const uint64_t mf = (uint64_t)((fb & 0x7FFFFFu) | 0x800000u);
  uint64_t V = sh >= 41 ? ~0ull : mf << sh;  // 2^-23 exactly would give 2^64
  {
    const __int128 E = (__int128)(((u128)1 << 116) - (u128)B * V);  // |E| < 2^96
    const int64_t Ep = (int64_t)(E >> 52);
    const uint64_t c = __umul64hi(V, (uint64_t)(Ep < 0 ? -Ep : Ep));
    V = Ep < 0 ? V - c : V + c;
  }
  {
    const __int128 E = (__int128)(((u128)1 << 116) - (u128)B * V);  // |E| < 2^75
    const int64_t Ep = (int64_t)(E >> 12);
    const uint64_t c = __umul64hi(V, (uint64_t)(Ep < 0 ? -Ep : Ep)) >> 40;
    V = Ep < 0 ? V - c : V + c;
  }
  uint64_t Q = (__umul64hi(Ma, V) << 2) | ((Ma * V) >> 62);
  uint64_t R = (Ma << 54) - Q * B;
  if ((int64_t)R < 0) {  // not reached when the bounds above hold
    R += B;
    --Q;
  }
  if (R >= B) {
    R -= B;
    ++Q;
  }
  if (R >= B) {  // not reached when the bounds above hold
    R -= B;
    ++Q;
  }
  rem_nz = R != 0;
  return Q;
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

// ---------------------------------------------------------------- wide integers

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


// ---------------------------------------------------------------- select helpers

// One warp: the bin of a kSelBins-bin histogram in shared memory that holds
// rank r (1-based), the count below that bin and the bin's own count, valid in
// every lane.  Lane l sums bins [64 l, 64 l + 64), a warp scan finds the lane
// whose range holds r, then the same over that lane's bins two at a time.
__device__ __forceinline__ void acc_scan_pick(const unsigned int *h, int64_t r, int &bin, int64_t &below,
                                              int64_t &cnt) {
  static_assert(kSelBins == 64 * 32, "64 bins per lane");
  const int lane = threadIdx.x & 31;
  int64_t s = 0;
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint4 *p = reinterpret_cast<const uint4 *>(h + 64 * lane + 4 * j);
    const uint4 q = *p;
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
  const uint2 pr = *p2;
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


// ---------------------------------------------------------------- phases

// First select digit: the top 12 + kbits bits of rel's pattern (exponent and
// kbits mantissa bits).  On the exact paths rel is 0 or lies in [2^elo,
// 2^(elo + octaves)), so the digit is offset to start there, with bin 0 for
// rel = 0; on the fp64 path it is the exponent field itself (bin 0 holds 0
// and the subnormals, bin 2047 inf and NaN).
struct AccKey {
  int kbits;  // mantissa bits in the digit
  int elo;    // lowest exponent of a non-zero rel (exact paths)
  int exact;  // offset layout with a zero bin
};

__device__ __forceinline__ int acc_key1(uint64_t rb, const AccKey &K) {
  if (!K.exact) return (int)(rb >> 52);
  if (rb == 0) return 0;
  const int64_t k = (int64_t)(rb >> (52 - K.kbits)) - ((int64_t)(1023 + K.elo) << K.kbits) + 1;
  return (int)min(max(k, (int64_t)1), (int64_t)kSelBins - 1);  // within range by construction
}

// Block-local view of the select, identical in every block (each derives it
// from the same global data in the same order).
struct AccSel {
  uint64_t pf[kAccTargets];   // prefix after the first digit; ~0 once a target is settled at 0
  int bin[kAccTargets];       // its first-digit bin
  int64_t rk[kAccTargets];    // rank still to find below it
  int64_t cnt[kAccTargets];   // samples in its bin
  int slot[kAccTargets];      // histogram shared by targets whose prefixes coincide
  int shift;                  // bits below the first digit
  int64_t m;                  // samples
};

// Exact pass over the block's range [lo, hi) of y and T on the narrow or
// wide grid: the sums into w, rel's patterns into `stage` (shared memory,
// when the range fits there) or relbits, rel's first digit
// into the block histogram h1 and rel into srel (fp64, in the thread's fixed
// order); `lost` when a value is off the wide grid.
template <bool kNarrow>
__device__ __forceinline__ void acc_exact_loop(const double *__restrict__ y, const double *__restrict__ T, int64_t lo,
                                               int64_t hi, int S, uint64_t *__restrict__ relbits, uint64_t *stage,
                                               uint64_t *w, unsigned int *h1, const AccKey &K, double &srel,
                                               bool &lost) {
  for (int64_t i0 = lo + threadIdx.x; i0 < hi; i0 += 4 * kAccBlock) {
    uint64_t yb[4], tb[4];  // four elements' loads in flight (a pattern of 0 is not a sample)
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t i = i0 + k * kAccBlock;
      yb[k] = i < hi ? (uint64_t)__double_as_longlong(__ldg(y + i)) : 0ull;
      tb[k] = i < hi ? (uint64_t)__double_as_longlong(__ldg(T + i)) : 0ull;
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t i = i0 + k * kAccBlock;
      uint64_t rb = ~0ull;  // not a sample
      if (acc_is_sample(yb[k])) {
        rb = kNarrow ? acc_exact_sample64(yb[k], tb[k], S, w) : acc_exact_sample(yb[k], tb[k], S, w, lost);
        atomicAdd(&h1[acc_key1(rb, K)], 1u);
        srel += __longlong_as_double((long long)rb);
      }
      if (i < hi) {
        if (stage)
          stage[i - lo] = rb;
        else
          relbits[i] = rb;
      }
    }
  }
}

// Counting sort of the block's samples by first digit: off = exclusive prefix
// sums of the block histogram h1, then each sample of the block's range (from
// `stage` when given, else relbits[lo, hi)) goes to
// sorted[lo + off[key] + (its place among the block's samples of that key)]
// (`cur`: kSelBins cursors of scratch).  Afterwards the samples of bin k lie
// at sorted[lo + off[k], lo + off[k] + h1[k]).
__device__ __forceinline__ void acc_block_sort(const uint64_t *__restrict__ relbits, const uint64_t *stage,
                                               uint64_t *__restrict__ sorted, int64_t lo, int64_t hi,
                                               const unsigned int *h1, unsigned int *off, unsigned int *cur,
                                               const AccKey &K) {
  __shared__ unsigned int wsum[kAccBlock / 32];
  constexpr int kPer = kSelBins / kAccBlock;  // bins per thread
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  unsigned int c[kPer], s = 0u;
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    c[j] = h1[threadIdx.x * kPer + j];
    s += c[j];
  }
  unsigned int inc = s;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const unsigned int o = __shfl_up_sync(0xffffffffu, inc, d);
    if (lane >= d) inc += o;
  }
  if (lane == 31) wsum[wid] = inc;
  __syncthreads();
  unsigned int wb = 0u;
  for (int v = 0; v < wid; ++v) wb += wsum[v];
  unsigned int run = wb + inc - s;
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    off[threadIdx.x * kPer + j] = run;
    cur[threadIdx.x * kPer + j] = run;
    run += c[j];
  }
  __syncthreads();
  if (stage) {
    for (int i = threadIdx.x; i < (int)(hi - lo); i += kAccBlock) {
      const uint64_t v = stage[i];
      if (v != ~0ull) sorted[lo + atomicAdd(&cur[acc_key1(v, K)], 1u)] = v;
    }
  } else {
    for (int64_t i0 = lo + threadIdx.x; i0 < hi; i0 += 4 * kAccBlock) {
      uint64_t v[4];  // four loads in flight
#pragma unroll
      for (int k = 0; k < 4; ++k) v[k] = i0 + k * kAccBlock < hi ? __ldcg(relbits + i0 + k * kAccBlock) : ~0ull;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (v[k] != ~0ull) sorted[lo + atomicAdd(&cur[acc_key1(v[k], K)], 1u)] = v[k];
    }
  }
  __syncthreads();
}

// Pick the digit of a histogram in shared memory (kSelBins bins) that holds
// rank r: bin, count below it, its count.  One warp; valid in every lane.
__device__ __forceinline__ void acc_pick1(const unsigned int *h, int64_t r, int &bin, int64_t &below, int64_t &cnt) {
  acc_scan_pick(h, r, bin, below, cnt);
}

// The r-th smallest (1-based) of the samples in `list` (c patterns) whose
// bits above `cur` equal `prefix`, by one block.  When they number at most
// kShort they are gathered into shared memory (`sh`) and ranked directly:
// the candidate with fewer than r smaller ones and at least r not larger;
// otherwise the remaining digits are settled from global memory, with `sh`
// as the digit histogram.
__device__ uint64_t acc_finish(const uint64_t *__restrict__ list, int64_t c, uint64_t prefix, int cur, int64_t r,
                               int64_t want, unsigned int *sh) {
  __shared__ uint64_t res;
  __shared__ int nsel;
  __shared__ int64_t pick[2];
  constexpr int kShort = kAccTargets * kSelBins / 2;
  if (want <= kShort) {
    uint64_t *ls = reinterpret_cast<uint64_t *>(sh);
    if (threadIdx.x == 0) {
      nsel = 0;
      res = 0ull;
    }
    __syncthreads();
    for (int64_t i0 = threadIdx.x; i0 < c; i0 += 4 * kAccBlock) {
      uint64_t v[4];  // four loads in flight
#pragma unroll
      for (int k = 0; k < 4; ++k) v[k] = i0 + k * kAccBlock < c ? __ldcg(list + i0 + k * kAccBlock) : ~0ull;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (i0 + k * kAccBlock < c && (v[k] >> cur) == prefix) {
          const int p = atomicAdd(&nsel, 1);
          if (p < kShort) ls[p] = v[k];
        }
    }
    __syncthreads();
    const int k = min(nsel, kShort);
    for (int i = threadIdx.x; i < k; i += kAccBlock) {
      const uint64_t v = ls[i];
      int64_t less = 0, leq = 0;
      for (int j = 0; j < k; ++j) {
        const uint64_t u = ls[j];
        less += u < v ? 1 : 0;
        leq += u <= v ? 1 : 0;
      }
      if (less < r && r <= leq) res = v;  // every finder holds the same value
    }
    __syncthreads();
    const uint64_t out = res;
    __syncthreads();
    return out;
  }
  while (cur > 0) {
    const int w = min(kSelBits, cur), lo = cur - w;
    const uint64_t dmask = (1ull << w) - 1;
    for (int i = threadIdx.x; i < kSelBins; i += kAccBlock) sh[i] = 0u;
    __syncthreads();
    for (int64_t i = threadIdx.x; i < c; i += kAccBlock) {
      const uint64_t v = __ldcg(list + i);
      if ((v >> cur) == prefix) atomicAdd(&sh[(int)((v >> lo) & dmask)], 1u);
    }
    __syncthreads();
    if (threadIdx.x < 32) {
      int bin;
      int64_t below, cnt;
      acc_scan_pick(sh, r, bin, below, cnt);
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
  return prefix;
}

// Sum of a double over the block's partials word `off` of every block, in a
// fixed order (thread j takes blocks j, j + blockDim, ...; then the block
// sum); valid in thread 0.
__device__ __forceinline__ double acc_fold_double(const uint64_t *part, int off, double *redd) {
  double s = 0.0;
  for (int b = threadIdx.x; b < (int)gridDim.x; b += kAccBlock)
    s += __longlong_as_double((long long)__ldcg(part + (int64_t)b * kAccPartW + off));
  return block_sum_fixed(s, redd);
}

// The r-th smallest (1-based) of the samples whose bits above `cur` equal
// `prefix`, c of them, found in the blocks' published segments of first-digit
// slot s (segs: nb x kAccTargets pairs of offset into `sorted` and length).
// By one block: at most kShort of them are gathered into shared memory and
// ranked directly, more are settled digit by digit over the segments.
__device__ uint64_t acc_finish_segs(const uint64_t *segs, const uint64_t *__restrict__ sorted, int nb, int s,
                                    uint64_t prefix, int cur, int64_t r, int64_t c, unsigned int *sh) {
  __shared__ uint64_t res;
  __shared__ int nsel;
  __shared__ int64_t pick[2];
  constexpr int kShort = kAccTargets * kSelBins / 2;
  auto each = [&](auto &&f) {  // every sample of the slot's segments, by the whole block
    for (int b = 0; b < nb; ++b) {
      const int64_t off = (int64_t)__ldcg(segs + 2 * (b * kAccTargets + s));
      const int64_t cnt = (int64_t)__ldcg(segs + 2 * (b * kAccTargets + s) + 1);
      for (int64_t i = threadIdx.x; i < cnt; i += kAccBlock) f(__ldcg(sorted + off + i));
    }
  };
  if (c <= kShort) {
    uint64_t *ls = reinterpret_cast<uint64_t *>(sh);
    if (threadIdx.x == 0) {
      nsel = 0;
      res = 0ull;
    }
    __syncthreads();
    each([&](uint64_t v) {
      if ((v >> cur) == prefix) {
        const int p = atomicAdd(&nsel, 1);
        if (p < kShort) ls[p] = v;
      }
    });
    __syncthreads();
    const int k = min(nsel, kShort);
    for (int i = threadIdx.x; i < k; i += kAccBlock) {
      const uint64_t v = ls[i];
      int64_t less = 0, leq = 0;
      for (int j = 0; j < k; ++j) {
        const uint64_t u = ls[j];
        less += u < v ? 1 : 0;
        leq += u <= v ? 1 : 0;
      }
      if (less < r && r <= leq) res = v;  // every finder holds the same value
    }
    __syncthreads();
    const uint64_t out = res;
    __syncthreads();
    return out;
  }
  while (cur > 0) {
    const int w = min(kSelBits, cur), lo = cur - w;
    const uint64_t dmask = (1ull << w) - 1;
    for (int i = threadIdx.x; i < kSelBins; i += kAccBlock) sh[i] = 0u;
    __syncthreads();
    each([&](uint64_t v) {
      if ((v >> cur) == prefix) atomicAdd(&sh[(int)((v >> lo) & dmask)], 1u);
    });
    __syncthreads();
    if (threadIdx.x < 32) {
      int bin;
      int64_t below, cnt;
      acc_scan_pick(sh, r, bin, below, cnt);
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
  return prefix;
}

// Exact totals to sums: fold the blocks' exact partials and write res[0] = m
// and, scaled by m 2^(2S), res[3..6] = sxx, syy, sxy, ssr (one each on
// threads 0..3).  One block.
__device__ __forceinline__ void acc_exact_totals(const AccArgs &a, uint64_t *redw) {
  __shared__ uint64_t tw[kAccWords];
  uint64_t w[kAccWords];
#pragma unroll
  for (int j = 0; j < kAccWords; ++j) w[j] = 0ull;
  for (int b = threadIdx.x; b < (int)gridDim.x; b += kAccBlock) {
    const uint64_t *p = a.part + (int64_t)b * kAccPartW + kPX;
    uint64_t o[kAccWords];
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) o[j] = __ldcg(p + j);
    acc_combine(w, o);
  }
  acc_block_combine(w, redw);
  if (threadIdx.x == 0)
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) tw[j] = w[j];
  __syncthreads();
  const int q = threadIdx.x;
  if (q >= 4) return;
#pragma unroll
  for (int j = 0; j < kAccWords; ++j) w[j] = tw[j];
  const uint64_t m = w[0];
  // |sum T| and its sign
  const bool tneg = (int64_t)w[4] < 0;
  const u128 st = ((u128)w[4] << 64) | w[3], sa = tneg ? (u128)0 - st : st;
  const uint64_t s0 = (uint64_t)sa, s1 = (uint64_t)(sa >> 64);
  uint64_t v[4], tmp[4];
  if (q == 0) {  // m sum Y^2 - (sum Y)^2
    mul64x192(m, w + 5, v);
    mul128x128(w[1], w[2], w[1], w[2], tmp);
    sub256(v, tmp);
  } else if (q == 1) {  // m sum T^2 - (sum T)^2
    mul64x192(m, w + 8, v);
    mul128x128(s0, s1, s0, s1, tmp);
    sub256(v, tmp);
  } else if (q == 2) {
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
    mul64x192(m, g, v);
    if (gneg) {
      uint64_t z[4] = {0, 0, 0, 0};
      sub256(z, v);
      v[0] = z[0];
      v[1] = z[1];
      v[2] = z[2];
      v[3] = z[3];
    }
    mul128x128(w[1], w[2], s0, s1, tmp);
    acc_add256(tmp, tmp[0], tmp[1], tmp[2], tmp[3]);  // 2 sum Y |sum T|
    if (tneg)
      acc_add256(v, tmp[0], tmp[1], tmp[2], tmp[3]);
    else
      sub256(v, tmp);
  } else {  // m sum D^2
    mul64x192(m, w + 11, v);
  }
  bool ok = true;  // every value here is below 2^227 in magnitude
  a.res[3 + q] = acc_i256_to_double(v, q == 2 ? -1 : 0, ok);
  if (q == 0) a.res[0] = (double)m;
}

// The samples of the block's segment for first-digit bin `bin` (the block's
// sorted range), visited by the whole block with eight loads in flight per
// thread.
template <class F>
__device__ __forceinline__ void acc_for_segment(const uint64_t *__restrict__ seg, int cnt, F &&visit) {
  for (int i0 = threadIdx.x; i0 < cnt; i0 += 8 * kAccBlock) {
    uint64_t v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = i0 + k * kAccBlock < cnt ? __ldcg(seg + i0 + k * kAccBlock) : ~0ull;
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (i0 + k * kAccBlock < cnt) visit(v[k]);
  }
}

// The whole accuracy computation of one call; a cooperative launch of at
// most as many blocks as fit at once.  Block b owns the elements [lo, hi).
__global__ void __launch_bounds__(kAccBlock) k_acc(AccArgs a) {
  extern __shared__ uint64_t stage_mem[];  // kAccStage patterns (dynamic): the block's rel values
  __shared__ __align__(16) unsigned int sh[kAccTargets * kSelBins];  // per-phase scratch
  __shared__ unsigned int bh1[kSelBins], bof1[kSelBins];  // the block's first-digit counts and offsets
  __shared__ unsigned long long red2[kAccBlock / 32 * 2];
  __shared__ double redd[kAccBlock / 32];
  __shared__ uint64_t redw[kAccBlock / 32 * kAccWords];
  __shared__ AccSel L, F;  // after the first digit; after the second (finishing blocks)
  __shared__ AccKey K;
  __shared__ int path[3];  // exact, narrow, S
  __shared__ double mean[2];
  int *err = reinterpret_cast<int *>(a.err);
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5, nb = gridDim.x;
  const int64_t n = a.n, stride = (int64_t)nb * kAccBlock, g0 = blockIdx.x * (int64_t)kAccBlock + tid;
  const int64_t chunk = (n + nb - 1) / nb, lo = min(n, chunk * blockIdx.x), hi = min(n, lo + chunk);
  uint64_t *mine = a.part + (int64_t)blockIdx.x * kAccPartW;
  const uint64_t *all = a.part;
  uint64_t *sorted = a.cand;  // each block's samples, sorted by first digit within its range

  // ---- range: the largest magnitude (high word of the largest sample y or
  // |T|) and smallest exponent over the samples' y and non-zero T.  (A NaN y
  // counts here, sending the call to the fp64 phases, which leave it out.)
  // The second-digit histograms, the first-digit totals and the list cursors
  // of the previous call are cleared here.
  for (int64_t i = g0; i < 2 * kSelBins; i += stride) a.hist1[i] = 0u;
  for (int64_t i = g0; i < kAccTargets * kSelBins; i += stride) a.hist2[i] = 0u;
  if (g0 == 0) *a.lost = 0;
  {
    unsigned int top = 0u, nmin = 0u;  // nmin: max of 2047 - biased exponent
    for (int64_t i0 = g0; i0 < n; i0 += 8 * stride) {
      uint2 yv[8], tv[8];  // eight elements' loads in flight (a pattern of 0 is not a sample)
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int64_t i = i0 + k * stride;
        yv[k] = i < n ? __ldg(reinterpret_cast<const uint2 *>(a.y) + i) : make_uint2(0u, 0u);
        tv[k] = i < n ? __ldg(reinterpret_cast<const uint2 *>(a.T) + i) : make_uint2(0u, 0u);
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const unsigned int yh = yv[k].y, th = tv[k].y & 0x7FFFFFFFu;
        if ((int)yh > 0 || (yh == 0u && yv[k].x != 0u)) {
          top = max(top, max(yh, th));
          nmin = max(nmin, 2047u - (yh >> 20));
          if (th | tv[k].x) nmin = max(nmin, 2047u - (th >> 20));
        }
      }
    }
    unsigned long long x = top, z = nmin;
    block_max2(x, z, red2);
    if (tid == 0) {
      mine[kPR] = x;
      mine[kPR + 1] = z;
    }
  }
  if (!grid_barrier(a.bar, err)) return acc_left(a);
  // the path: exact when the values are finite, n < 2^32 (the integer widths
  // hold any count below it) and Emax is in [kAccEmaxLo, kAccEmaxHi]; narrow
  // (64-bit integers) when every exponent is within 10 of Emax
  {
    unsigned long long x = 0ull, z = 0ull;
    for (int b = tid; b < nb; b += kAccBlock) {
      x = max(x, (unsigned long long)__ldcg(all + (int64_t)b * kAccPartW + kPR));
      z = max(z, (unsigned long long)__ldcg(all + (int64_t)b * kAccPartW + kPR + 1));
    }
    block_max2(x, z, red2);
    if (tid == 0) {
      const int E = (int)(x >> 20) - 1023, Emin = 2047 - (int)z - 1023;  // no sample: nothing to sum
      const bool ex = x < 0x7FF00000ull && n < ((int64_t)1 << 32) && (z == 0 || (E >= kAccEmaxLo && E <= kAccEmaxHi));
      path[0] = ex;
      path[1] = ex && E - Emin <= 10;
      path[2] = (E - Emin <= 10 ? 62 : kAccGrid) - E;
      // rel's exponents on the exact paths: [-63, 12] on the narrow grid
      // (|D| < 2^64 and y >= 2^52 grid units, a non-zero |D| at least one),
      // [-79, 80] on the wide one (|D| < 2^80, y at least one unit, below 2^79)
      K.exact = 1;
      K.kbits = path[1] ? 4 : 3;
      K.elo = path[1] ? -63 : -79;
    }
    for (int i = tid; i < kSelBins; i += kAccBlock) bh1[i] = 0u;
    __syncthreads();
  }

  // ---- exact: sums, rel and its first digit on the grid; the block's
  // samples sorted by first digit
  bool fp64 = path[0] == 0;
  if (!fp64) {
    uint64_t w[kAccWords];
#pragma unroll
    for (int j = 0; j < kAccWords; ++j) w[j] = 0ull;
    double srel = 0.0;
    bool lost = false;
    uint64_t *stage = hi - lo <= kAccStage ? stage_mem : nullptr;
    if (path[1])
      acc_exact_loop<true>(a.y, a.T, lo, hi, path[2], a.relbits, stage, w, bh1, K, srel, lost);
    else
      acc_exact_loop<false>(a.y, a.T, lo, hi, path[2], a.relbits, stage, w, bh1, K, srel, lost);
    if (__syncthreads_or(lost) && tid == 0) atomicOr(a.lost, 1);
    acc_block_sort(a.relbits, stage, sorted, lo, hi, bh1, bof1, sh, K);
    for (int i = tid; i < kSelBins; i += kAccBlock) {
      const unsigned int c = bh1[i];
      if (c) atomicAdd(a.hist1 + i, c);
    }
    srel = block_sum_fixed(srel, redd);
    acc_block_combine(w, redw);
    if (tid == 0) {
      mine[kPC] = w[0];
      mine[kPQ] = (uint64_t)__double_as_longlong(srel);
#pragma unroll
      for (int j = 0; j < kAccWords; ++j) mine[kPX + j] = w[j];
    }
    if (!grid_barrier(a.bar, err)) return acc_left(a);
    fp64 = __ldcg(a.lost) != 0;  // a value off the wide grid: redo the call in fp64
  }

  // ---- fp64: rel and its first digit, the block's samples sorted by it,
  // means, then centred moments, each in a fixed order
  if (fp64) {
    if (tid == 0) {
      K.exact = 0;
      K.kbits = 0;
      K.elo = 0;
    }
    for (int i = tid; i < kSelBins; i += kAccBlock) bh1[i] = 0u;
    __syncthreads();
    double c = 0.0, sy = 0.0, st = 0.0, srel = 0.0;
    uint64_t cnt = 0;
    for (int64_t i = lo + tid; i < hi; i += kAccBlock) {
      const double yv = a.y[i], tv = a.T[i];
      uint64_t bits = ~0ull;
      if (yv > 0.0) {
        c += 1.0;
        ++cnt;
        sy += yv;
        st += tv;
        bits = (uint64_t)__double_as_longlong(__ddiv_rn(fabs(__dsub_rn(tv, yv)), yv));
        atomicAdd(&bh1[(int)(bits >> 52)], 1u);
        srel += __longlong_as_double((long long)bits);
      }
      a.relbits[i] = bits;
    }
    __syncthreads();
    acc_block_sort(a.relbits, nullptr, sorted, lo, hi, bh1, bof1, sh, K);
    for (int i = tid; i < kSelBins; i += kAccBlock) {
      const unsigned int h = bh1[i];
      if (h) atomicAdd(a.hist1 + kSelBins + i, h);
    }
    const double A = block_sum_fixed(c, redd), B = block_sum_fixed(sy, redd), C = block_sum_fixed(st, redd);
    srel = block_sum_fixed(srel, redd);
#pragma unroll
    for (int d = 16; d; d >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, d);
    __syncthreads();
    if (lane == 0) redw[wid] = cnt;
    __syncthreads();
    if (tid == 0) {
      uint64_t tc = 0;
      for (int v = 0; v < kAccBlock / 32; ++v) tc += redw[v];
      double *p = reinterpret_cast<double *>(mine);
      mine[kPC] = tc;
      mine[kPQ] = (uint64_t)__double_as_longlong(srel);
      p[kPS] = A;
      p[kPS + 1] = B;
      p[kPS + 2] = C;
    }
    if (!grid_barrier(a.bar, err)) return acc_left(a);
    const double s0 = acc_fold_double(all, kPS, redd), s1 = acc_fold_double(all, kPS + 1, redd),
                 s2 = acc_fold_double(all, kPS + 2, redd);
    if (tid == 0) {
      mean[0] = s0 > 0 ? s1 / s0 : 0.0;
      mean[1] = s0 > 0 ? s2 / s0 : 0.0;
    }
    __syncthreads();
    const double my = mean[0], mt = mean[1];
    double sxx = 0.0, syy = 0.0, sxy = 0.0, ssr = 0.0;
    for (int64_t i = lo + tid; i < hi; i += kAccBlock) {
      const double yv = a.y[i], tv = a.T[i];
      if (yv > 0.0) {
        const double dy = yv - my, dt = tv - mt, e = yv - tv;
        sxx += dy * dy;
        syy += dt * dt;
        sxy += dy * dt;
        ssr += e * e;
      }
    }
    const double v0 = block_sum_fixed(sxx, redd), v1 = block_sum_fixed(syy, redd), v2 = block_sum_fixed(sxy, redd),
                 v3 = block_sum_fixed(ssr, redd);
    if (tid == 0) {
      double *p = reinterpret_cast<double *>(mine);
      p[kPM] = v0;
      p[kPM + 1] = v1;
      p[kPM + 2] = v2;
      p[kPM + 3] = v3;
    }
    if (!grid_barrier(a.bar, err)) return acc_left(a);
  }

  // ---- first digit: the sample count (the histogram's total), then each
  // target's bin (every block)
  {
    const unsigned int *h1 = a.hist1 + (fp64 ? kSelBins : 0);
    for (int i = tid; i < kSelBins; i += kAccBlock) sh[i] = __ldcg(h1 + i);
    __syncthreads();
    if (wid == 0) {
      unsigned long long c = 0ull;
      for (int i = lane; i < kSelBins; i += 32) c += sh[i];
#pragma unroll
      for (int d = 16; d; d >>= 1) c += __shfl_xor_sync(0xffffffffu, c, d);
      if (lane == 0) {
        const int64_t m = (int64_t)c;
        L.m = m;
        L.shift = 52 - K.kbits;
        for (int t = 0; t < kAccTargets; ++t) {
          const int64_t q = t == 0 ? 50 : t == 1 ? 90 : 99;
          L.rk[t] = (q * m + 99) / 100;
        }
      }
    }
    __syncthreads();
    int bin = 0;
    int64_t below = 0, c1 = 0;
    if (wid < kAccTargets && L.m > 0) acc_pick1(sh, L.rk[wid], bin, below, c1);
    if (wid < kAccTargets && lane == 0) {
      L.bin[wid] = bin;
      if (L.m == 0 || (K.exact && bin == 0)) {
        L.pf[wid] = ~0ull;  // settled: rel = 0 (or no sample)
        L.cnt[wid] = 0;
      } else {
        L.pf[wid] = K.exact ? (uint64_t)(bin - 1) + ((uint64_t)(1023 + K.elo) << K.kbits) : (uint64_t)bin;
        L.rk[wid] -= below;
        L.cnt[wid] = c1;
      }
    }
    __syncthreads();
    if (tid == 0)
      for (int t = 0; t < kAccTargets; ++t) {  // targets in the same bin share one second-digit histogram
        int s = t;
        for (int u = t - 1; u >= 0; --u)
          if (L.pf[u] == L.pf[t]) s = L.slot[u];
        L.slot[t] = s;
      }
    __syncthreads();
  }

  // ---- second digit: each block histograms the next 11 bits of its samples
  // in the targets' first-digit bins (its sorted segments), keeping each
  // bin's first kAccBucket samples in a bucket and publishing where its
  // segments lie
  {
    const int lo2 = L.shift - kSelBits;
    for (int t = 0; t < kAccTargets; ++t) {
      if (L.slot[t] != t || L.pf[t] == ~0ull) continue;  // the same in every block
      const int b = L.bin[t];
      unsigned int *h2 = a.hist2 + t * kSelBins;
      uint64_t *bk = a.bucket + (int64_t)t * kSelBins * kAccBucket;
      acc_for_segment(sorted + lo + bof1[b], (int)bh1[b], [&](uint64_t v) {
        const int d = (int)((v >> lo2) & (uint64_t)(kSelBins - 1));
        const unsigned int p = atomicAdd(h2 + d, 1u);
        if (p < kAccBucket) bk[d * kAccBucket + p] = v;  // the bin's first samples, kept for the finish
      });
      if (tid == 0) {
        a.segs[2 * (blockIdx.x * kAccTargets + t)] = (uint64_t)(lo + bof1[b]);
        a.segs[2 * (blockIdx.x * kAccTargets + t) + 1] = bh1[b];
      }
    }
  }
  if (!grid_barrier(a.bar, err)) return acc_left(a);

  // ---- finish: block t picks target t's second digit and ranks its
  // candidates (from the bin's bucket, or from every block's segment when
  // the bin outgrew its bucket); other blocks form the totals
  uint64_t *pct = reinterpret_cast<uint64_t *>(a.res + 8);
  for (int t = blockIdx.x; t < kAccTargets; t += nb) {
    uint64_t r = 0ull;
    if (L.pf[t] != ~0ull) {
      const int s = L.slot[t];
      for (int i = tid; i < kSelBins; i += kAccBlock) sh[i] = __ldcg(a.hist2 + s * kSelBins + i);
      __syncthreads();
      if (wid == 0) {
        int bin;
        int64_t below, c2;
        acc_pick1(sh, L.rk[t], bin, below, c2);
        if (lane == 0) {
          F.pf[t] = (L.pf[t] << kSelBits) | (uint64_t)bin;
          F.rk[t] = L.rk[t] - below;
          F.cnt[t] = c2;
        }
      }
      __syncthreads();
      const int cur = L.shift - kSelBits;
      if (F.cnt[t] <= kAccBucket)
        r = acc_finish(a.bucket + ((int64_t)s * kSelBins + (int64_t)(F.pf[t] & (kSelBins - 1))) * kAccBucket,
                       F.cnt[t], F.pf[t], cur, F.rk[t], F.cnt[t], sh);
      else
        r = acc_finish_segs(a.segs, sorted, nb, s, F.pf[t], cur, F.rk[t], F.cnt[t], sh);
    }
    if (tid == 0) pct[t] = r;
    __syncthreads();
  }
  if (blockIdx.x == (kAccTargets % nb)) {
    if (!fp64) {
      acc_exact_totals(a, redw);
    } else {
      double v[4];
      for (int j = 0; j < 4; ++j) v[j] = acc_fold_double(all, kPM + j, redd);
      if (tid == 0) {
        a.res[0] = (double)L.m;
        for (int j = 0; j < 4; ++j) a.res[3 + j] = v[j];
      }
    }
  }
  if (blockIdx.x == ((kAccTargets + 1) % nb)) {
    __syncthreads();
    const double sr = acc_fold_double(all, kPQ, redd);
    if (tid == 0) a.res[7] = sr;
  }
}

// Barrier self-test: the last block leaves without arriving, so the others'
// wait at the barrier runs out and sets the error word.
__global__ void k_barrier_probe(unsigned int *bar, int *err) {
  if (blockIdx.x == gridDim.x - 1) return;
  grid_barrier(bar, err);
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
