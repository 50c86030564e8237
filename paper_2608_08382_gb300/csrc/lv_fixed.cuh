// Exact integer fixed-point arithmetic for Eq. 1 on the integer pipes.
//
// GB300 issues double-precision FMAs at 1/64 of the FP32 rate and converts
// integers to double on the same slow pipe, so the per-request and per-batch
// arithmetic of the latency model is carried out in 128-bit two's-complement
// integers instead: every coefficient a_k is an exact integer multiple of a
// per-segment power of two 2^E, the features p, c, p^2, S1.. are integers, so
// a_k * x_k is an exact integer product and the whole linear form is an exact
// integer sum.  The single rounding to double happens at the end, from bits.
#pragma once

#include <cstdint>

namespace lv {

struct i128 {
  uint64_t lo;
  uint64_t hi;  // two's complement high word
};

__host__ __device__ __forceinline__ i128 mk128(uint64_t lo, uint64_t hi) {
  i128 r;
  r.lo = lo;
  r.hi = hi;
  return r;
}

__host__ __device__ __forceinline__ i128 add128(i128 a, i128 b) {
  i128 r;
  r.lo = a.lo + b.lo;
  r.hi = a.hi + b.hi + (r.lo < a.lo ? 1ull : 0ull);
  return r;
}

__host__ __device__ __forceinline__ i128 neg128(i128 a) {
  i128 r;
  r.lo = ~a.lo + 1ull;
  r.hi = ~a.hi + (r.lo == 0 ? 1ull : 0ull);
  return r;
}

__host__ __device__ __forceinline__ bool is_neg128(i128 a) { return (int64_t)a.hi < 0; }

// Low 128 bits of A * x for 0 <= x < 2^32 (exact when the true product fits).
__device__ __forceinline__ i128 mul128_u32(i128 A, uint32_t x) {
  const uint64_t p0 = (uint64_t)(uint32_t)A.lo * x;          // bits   0..63
  const uint64_t p1 = (uint64_t)(uint32_t)(A.lo >> 32) * x;  // bits  32..95
  const uint64_t p2 = (uint64_t)(uint32_t)A.hi * x;          // bits  64..127
  const uint32_t p3 = (uint32_t)(A.hi >> 32) * x;            // bits  96..127 (low half)
  i128 r;
  r.lo = p0 + (p1 << 32);
  const uint64_t c = (r.lo < p0) ? 1ull : 0ull;
  r.hi = (p1 >> 32) + p2 + ((uint64_t)p3 << 32) + c;
  return r;
}

// Low 128 bits of A * x for 0 <= x < 2^64.
__device__ __forceinline__ i128 mul128_u64(i128 A, uint64_t x) {
  i128 lo = mul128_u32(A, (uint32_t)x);
  const uint32_t xh = (uint32_t)(x >> 32);
  if (xh == 0) return lo;
  i128 hi = mul128_u32(A, xh);
  i128 sh;
  sh.lo = hi.lo << 32;
  sh.hi = (hi.hi << 32) | (hi.lo >> 32);
  return add128(lo, sh);
}

// 128-bit left shift, 0 <= s < 128.
__host__ __device__ __forceinline__ i128 shl128(uint64_t lo, uint64_t hi, int s) {
  i128 r;
  if (s == 0) {
    r.lo = lo;
    r.hi = hi;
  } else if (s < 64) {
    r.hi = (hi << s) | (lo >> (64 - s));
    r.lo = lo << s;
  } else {
    r.hi = lo << (s - 64);
    r.lo = 0;
  }
  return r;
}

// Result of rounding a fixed-point value to double: the double itself and the
// rounded value as +-m * 2^ex (m <= 2^53 including the implicit bit), which the
// tenant accumulator re-expands exactly.
struct Rounded {
  double d;
  uint64_t m;
  int ex;
  bool neg;
};

// Round V * 2^E to the nearest double, ties to even.  The caller guarantees the
// exponent stays in the normal range (-1022 <= E and E + 127 <= 1023).
__device__ __forceinline__ Rounded fix_to_double(i128 V, int E) {
  Rounded r;
  r.neg = is_neg128(V);
  if (r.neg) V = neg128(V);
  if ((V.hi | V.lo) == 0) {
    r.d = 0.0;
    r.m = 0;
    r.ex = 0;
    r.neg = false;
    return r;
  }
  const int lz = V.hi ? __clzll((long long)V.hi) : 64 + __clzll((long long)V.lo);
  const i128 N = shl128(V.lo, V.hi, lz);           // leading one at bit 127
  uint64_t m = N.hi >> 11;                           // 53 significant bits
  const uint64_t rb = (N.hi >> 10) & 1ull;
  const uint64_t st = ((N.hi & 0x3FFull) | N.lo) != 0 ? 1ull : 0ull;
  m += rb & (st | (m & 1ull));                       // may carry to 2^53
  const int ex = 127 - lz + E;                       // exponent of the leading bit
  const uint64_t bits = ((uint64_t)(ex + 1023) << 52) + (m - (1ull << 52));
  r.d = __longlong_as_double((long long)(bits | ((uint64_t)r.neg << 63)));
  r.m = m;
  r.ex = ex - 52;                                    // value = m * 2^(ex-52)
  return r;
}

// Same as fix_to_double for the common case 2^64 <= V < 2^127 (V > 0, high
// word non-zero): no sign handling and a branch-free normalisation.
__device__ __forceinline__ Rounded fix_to_double_pos(i128 V, int E) {
  if ((int64_t)V.hi <= 0) return fix_to_double(V, E);
  const int lz = __clzll((long long)V.hi);  // 1..63
  const uint64_t top = (V.hi << lz) | (V.lo >> (64 - lz));
  const uint64_t rest = V.lo << lz;
  uint64_t m = top >> 11;
  const uint64_t rb = (top >> 10) & 1ull;
  const uint64_t st = ((top & 0x3FFull) | rest) != 0 ? 1ull : 0ull;
  m += rb & (st | (m & 1ull));
  const int ex = 127 - lz + E;
  Rounded r;
  r.d = __longlong_as_double((long long)(((uint64_t)(ex + 1023) << 52) + (m - (1ull << 52))));
  r.m = m;
  r.ex = ex - 52;
  r.neg = false;
  return r;
}

// V * 2^E rounded to the nearest double (ties to even) for the common
// magnitude 2^64 <= V < 2^96 (v3 = 0, v2 != 0; the caller checks): the
// leading word is v2.  m is the rounded significand (2^52 <= m <= 2^53) and
// ex2 its exponent: the result equals m * 2^ex2.
__device__ __forceinline__ double round96(uint32_t v0, uint32_t v1, uint32_t v2, int E, uint64_t &m, int &ex2) {
  const int s = __clz(v2);
  const uint32_t t2 = __funnelshift_l(v1, v2, s), t1 = __funnelshift_l(v0, v1, s), t0 = v0 << s;
  uint32_t mhi = t2 >> 11, mlo = __funnelshift_r(t1, t2, 11);
  const uint32_t inc = ((t1 >> 10) & 1u) & ((((t1 & 0x3ffu) | t0) != 0u ? 1u : 0u) | (mlo & 1u));
  mlo += inc;
  mhi += mlo < inc ? 1u : 0u;
  const int ex = 95 - s + E;  // exponent of the leading bit
  m = ((uint64_t)mhi << 32) | mlo;
  ex2 = ex - 52;
  // bits = (ex + 1022) 2^52 + m: m's implicit bit (2^52, or 2^53 after a carry) completes the exponent
  return __hiloint2double((int)(((uint32_t)(ex + 1022) << 20) + mhi), (int)mlo);
}

// Exact double -> fixed point at 2^E, rounded to nearest (ties to even) when
// the double has bits below 2^E.  Sets *ovf when the value needs >= 2^125.
__host__ __device__ __forceinline__ i128 double_to_fix(double x, int E, bool *ovf) {
  uint64_t b;
#ifdef __CUDA_ARCH__
  b = (uint64_t)__double_as_longlong(x);
#else
  __builtin_memcpy(&b, &x, 8);
#endif
  const bool neg = (b >> 63) != 0;
  const int be = (int)((b >> 52) & 0x7FF);
  uint64_t m = b & ((1ull << 52) - 1);
  int ex;
  if (be == 0) {
    ex = -1074;
  } else {
    m |= 1ull << 52;
    ex = be - 1075;
  }
  i128 r = mk128(0, 0);
  if (be == 0x7FF) {
    *ovf = true;
    return r;
  }
  if (m == 0) return r;
  const int sh = ex - E;
  if (sh >= 0) {
    if (sh > 125 - 53) {
      *ovf = true;
      return r;
    }
    r = shl128(m, 0, sh);
  } else {
    const int rs = -sh;
    if (rs > 60) {
      // below half an LSB: rounds to zero (m < 2^53 <= 2^(rs-1))
      return r;
    }
    uint64_t q = m >> rs;
    const uint64_t rem = m & ((1ull << rs) - 1);
    const uint64_t half = 1ull << (rs - 1);
    if (rem > half || (rem == half && (q & 1ull))) ++q;
    r = mk128(q, 0);
  }
  return neg ? neg128(r) : r;
}

}  // namespace lv
