// Device code shared by the LLMVisor kernels (sm_103a): model parameters, the
// merge-path partition, exact fixed-point evaluation of Eq. 1 and of the
// per-request shares, exact tenant accumulation, and the small kernels around
// them.  The request-streaming kernels themselves are in lv_warp.cuh.
#pragma once

#include <cstddef>
#include <cstdint>

#include "lv_fixed.cuh"

namespace lv {

constexpr int kBlock = 256;                        // threads per CTA of the small kernels
constexpr int kHotMax = 512;                       // tenants kept in shared memory per CTA
constexpr int kNK = 256;                           // per-batch constants cached in shared memory for n <= kNK
constexpr int64_t kPMaxFix = 1ll << 24;            // p beyond this uses the fp64 share path
constexpr int kTenLsb = -72;                       // tenant totals: shares rounded to 2^-72 s, summed exactly

// Bits of the sticky status word: invalid input data; a fit feature beyond
// the exact range (bit 2 is reserved).
constexpr int kStatusData = 1;
constexpr int kStatusOverflow = 4;
constexpr int kStatusTimeout = 8;  // a bounded wait inside a kernel ran out

struct SegFix {
  i128 A1, A2, A3;   // exact a_k * 2^-E
  i128 B, A4;        // beta and a4 at 2^E (rounded to nearest)
  i128 A13;          // A1 + A3: the p-terms of a decode request (p = 1)
  uint64_t lim[4];   // exact T path valid when S1, S2, S3, n^2 <= lim[0..3]
  int E;
  int a2_narrow;     // 1: 0 <= A2 < 2^64 (64-bit multiply suffices)
  int t_narrow;      // 1: B, A1..A4 all in [0, 2^96) (eq1_fast applies)
  int pad;
};

struct KEntry {
  double q;    // fl(beta / n)
  double a4n;  // fl(a4 * n)
  i128 kf;     // fl(q + a4n) at 2^E, or kKSlowHi in the high word when it does not fit
};

// High word of KEntry::kf marking a constant outside the fixed-point range
// (|K| < 2^125 otherwise, so this value never occurs).
constexpr uint64_t kKSlowHi = 0x8000000000000000ull;

struct ModelP {
  double coef[4][5];
  int64_t split[2];
  SegFix fx[4];
  const KEntry *ktab;  // [4][nk + 1]
  int nk;
  int fixed;           // 1: integer fixed-point path
};

constexpr int kFitMaxY = 4;             // latency vectors fitted per pass
constexpr int kFitYLsb = -100;          // X^T y fixed point: y rounded to 2^-100 s
constexpr int64_t kFitFeatMax = 1ll << 48;

constexpr int kFitYYLsb = 2 * kFitYLsb + 64;  // y'y: floor(Y^2 / 2^64) summed, LSB 2^-136 s^2

// Entries per group: 15 Gram pairs (a <= b), 5 X^T y per y, 1 y'y per y, 1 flag.
__host__ __device__ constexpr int fit_entries(int n_y) { return 16 + 6 * n_y; }

struct FitAcc {
  uint64_t w[4];  // 256-bit two's complement (Gram: low 128 bits; flag: w[0])
};

struct FitArgs {
  const double *y;  // [n_y][n_batch]
  int n_y;
  FitAcc *partial;  // [gridDim.x][4 * fit_entries(n_y)]
};

__device__ __forceinline__ void acc_add256(uint64_t *w, uint64_t a0, uint64_t a1, uint64_t a2, uint64_t a3) {
  uint64_t s = w[0] + a0;
  uint64_t c = s < a0 ? 1ull : 0ull;
  w[0] = s;
  s = w[1] + a1;
  uint64_t c2 = s < a1 ? 1ull : 0ull;
  s += c;
  c2 |= (s < c) ? 1ull : 0ull;
  w[1] = s;
  s = w[2] + a2;
  uint64_t c3 = s < a2 ? 1ull : 0ull;
  s += c2;
  c3 |= (s < c2) ? 1ull : 0ull;
  w[2] = s;
  w[3] = w[3] + a3 + c3;
}

// Exact y * 2^100 as a signed 128-bit integer (round to nearest even below 2^-100).
__device__ __forceinline__ i128 y_fixed(double y, bool *ovf) {
  return double_to_fix(y, kFitYLsb, ovf);
}

// One batch into the owner's accumulator.  x[0..4] = 1, S1, S2, S3, n^2.
__device__ __forceinline__ void fit_owner_add(FitAcc &acc, int e, int n_y, const int64_t x[5], const double *yv,
                                              int64_t nb, int64_t gb, bool s1_ne_s3, int *bad) {
  if (e < 15) {
    // Gram pair (a, b), a <= b, in row order
    int a = 0, r = e;
    while (r >= 5 - a) {
      r -= 5 - a;
      ++a;
    }
    const int b = a + r;
    const uint64_t u = (uint64_t)x[a], v = (uint64_t)x[b];
    acc_add256(acc.w, u * v, __umul64hi(u, v), 0, 0);
  } else if (e < 15 + 5 * n_y) {
    const int col = (e - 15) % 5, k = (e - 15) / 5;
    bool ovf = false;
    const i128 Y = y_fixed(yv[k * nb + gb], &ovf);
    if (ovf) *bad = 1;
    const bool neg = is_neg128(Y);
    const i128 M = neg ? neg128(Y) : Y;
    const uint64_t xv = (uint64_t)x[col];
    // |Y| * x as 192 bits
    const uint64_t p0 = M.lo * xv, p1 = __umul64hi(M.lo, xv);
    const uint64_t q0 = M.hi * xv, q1 = __umul64hi(M.hi, xv);
    uint64_t w0 = p0, w1 = p1 + q0, w2 = q1 + (w1 < p1 ? 1ull : 0ull), w3 = 0;
    if (neg) {
      w0 = ~w0;
      w1 = ~w1;
      w2 = ~w2;
      w3 = ~w3;
      w0 += 1;
      if (w0 == 0) {
        w1 += 1;
        if (w1 == 0) {
          w2 += 1;
          if (w2 == 0) w3 += 1;
        }
      }
    }
    acc_add256(acc.w, w0, w1, w2, w3);
  } else if (e < 15 + 6 * n_y) {
    // y'y: Y^2 (below 2^250) shifted right by 64 bits; a sum of integers, so
    // order independent, with an error below n * 2^-136 s^2
    const int k = e - 15 - 5 * n_y;
    bool ovf = false;
    i128 Y = y_fixed(yv[k * nb + gb], &ovf);
    if (ovf) *bad = 1;
    if (is_neg128(Y)) Y = neg128(Y);
    const uint64_t l = Y.lo, h = Y.hi;
    const uint64_t ll1 = __umul64hi(l, l), hl0 = h * l, hl1 = __umul64hi(h, l);
    const uint64_t hh0 = h * h, hh1 = __umul64hi(h, h);
    // words 1..3 of l*l + 2^64 * 2*h*l + 2^128 * h*h (word 0 is dropped)
    uint64_t w[4] = {ll1, hh0, hh1, 0};
    acc_add256(w, hl0, hl1, 0, 0);
    acc_add256(w, hl0, hl1, 0, 0);
    acc_add256(acc.w, w[0], w[1], w[2], 0);
  } else {
    if (s1_ne_s3) acc.w[0] |= 1ull;
  }
}

// First batch of a tile and its first request.
struct TilePart {
  int64_t b;
  int64_t r;
};

struct TileArgs {
  const int32_t *p, *c, *ph, *ten;
  const int64_t *off;
  int64_t n_req, n_batch;
  const TilePart *part;  // [n_tiles + 1]
  int64_t n_tiles;
  int64_t D;             // merge positions per tile
  double *T, *share;
  float *T32, *share32;  // fp32 variant (M_F32): T and shares as float, or null
  int64_t *bfeat;   // [5][n_batch] or null
  uint8_t *bseg;    // [n_batch] or null
  unsigned long long *ten_pend;  // [n_tenants][4] 32-bit limbs in 64-bit words, or null
  int32_t n_tenants, H;
  int *status;
  ModelP mp;
  FitArgs fit;
  unsigned long long *ctr;      // warp tiles handed out so far (zeroed before the launch)
  unsigned long long *jumbo_n;  // batches queued for k_jumbo (zeroed before the launch)
  int64_t *jumbo;               // [jumbo_cap] queued batch indices
  int64_t jumbo_cap;
};

__device__ __forceinline__ void flag(int *status, int bit) {
  if (status) atomicOr(status, bit);
}

__device__ __forceinline__ int64_t clampi(int64_t v, int64_t lo, int64_t hi) {
  return v < lo ? lo : (v > hi ? hi : v);
}

// ---------------------------------------------------------------- merge-path partition

// part[k] = {b, off[b]} for the first batch b with b + off[b] >= k*D, for
// k in [0, n_tiles); part[n_tiles] = {n_batch, n_req}.  Batch b writes the k in
// (f(b-1)/D, f(b)/D], so every entry is written once by a coalesced pass.
__global__ void k_partition(const int64_t *__restrict__ off, int64_t n_batch, int64_t n_req, int64_t n_tiles,
                            int64_t D, TilePart *__restrict__ part, int *status) {
  int bad = 0;
  for (int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; b <= n_batch;
       b += (int64_t)gridDim.x * blockDim.x) {
    const int64_t raw = __ldg(off + b);
    const int64_t ob = clampi(raw, 0, n_req);
    int64_t kmin;
    if (b == 0) {
      if (raw != 0) bad = 1;
      kmin = 0;
    } else {
      const int64_t rp = __ldg(off + b - 1);
      if (rp > raw) bad = 1;
      kmin = (b - 1 + clampi(rp, 0, n_req)) / D + 1;
    }
    int64_t kmax = (b + ob) / D;
    if (b == n_batch) {
      if (raw != n_req) bad = 1;
      kmax = n_tiles;
    }
    if (kmin < 0) kmin = 0;
    if (kmax > n_tiles) kmax = n_tiles;
    for (int64_t k = kmin; k <= kmax; ++k) {
      TilePart tp;
      tp.b = b;
      tp.r = ob;
      part[k] = tp;
    }
  }
  if (bad) flag(status, kStatusData);
}

// ---------------------------------------------------------------- batch sums

struct Sums {
  int64_t s1, s2, s3;
  int32_t ph;
};

// ---------------------------------------------------------------- model arithmetic

struct BatchAgg {
  int64_t s1, s2, s3, n;
  int prefill;
};

// Segment of a batch (phase: any prefill request; regime: S1 >= split[phase]).
__device__ __forceinline__ int segment_of(const ModelP &mp, const BatchAgg &g) {
  if (g.n == 0) return 0;
  const int ph = g.prefill ? 1 : 0;
  return ph * 2 + (g.s1 >= mp.split[ph] ? 1 : 0);
}

// Eq. 1 left to right in double, no contraction (same rounding sequence as a
// plain sequential evaluation).
__device__ __forceinline__ double eq1_fp64(const double *k, const BatchAgg &g) {
  if (g.n == 0) return 0.0;
  double T = k[0];
  T = __dadd_rn(T, __dmul_rn(k[1], (double)g.s1));
  T = __dadd_rn(T, __dmul_rn(k[2], (double)g.s2));
  T = __dadd_rn(T, __dmul_rn(k[3], (double)g.s3));
  T = __dadd_rn(T, __dmul_rn(k[4], (double)(g.n * g.n)));
  return T;
}

// Eq. 1 exactly in fixed point, one rounding; falls back to fp64 outside the
// exact range.  Once per batch, so kept out of line.
__device__ __noinline__ double eq1_fix(const ModelP &mp, int s, const BatchAgg &g) {
  if (g.n == 0) return 0.0;
  const SegFix &f = mp.fx[s];
  const uint64_t F4 = (uint64_t)g.n * (uint64_t)g.n;
  if ((uint64_t)g.s1 > f.lim[0] || (uint64_t)g.s2 > f.lim[1] || (uint64_t)g.s3 > f.lim[2] || F4 > f.lim[3] ||
      g.n > 0x7fffffffll)
    return eq1_fp64(mp.coef[s], g);
  i128 V = f.B;
  V = add128(V, mul128_u64(f.A1, (uint64_t)g.s1));
  V = add128(V, mul128_u64(f.A2, (uint64_t)g.s2));
  V = add128(V, mul128_u64(f.A3, (uint64_t)g.s3));
  V = add128(V, mul128_u64(f.A4, F4));
  return fix_to_double(V, f.E).d;
}

// Eq. 1 in fixed point for the common case: every coefficient in [0, 2^96)
// (t_narrow), each product A_k S_k below 2^96 and the sum in [2^64, 2^96);
// 64x64-bit products with the coefficients' high words folded in, and the
// leading-word rounding.  False when any of these does not hold (the caller
// then takes eq1_fix, which gives the same value wherever this one applies).
__device__ __forceinline__ bool eq1_fast(const SegFix &f, const BatchAgg &g, double *T) {
  if (!f.t_narrow || g.n == 0 || g.n > 0x7fffffffll) return false;
  uint64_t lo = f.B.lo, hi = f.B.hi;
  bool ok = true;
  const i128 A[4] = {f.A1, f.A2, f.A3, f.A4};
  const uint64_t S[4] = {(uint64_t)g.s1, (uint64_t)g.s2, (uint64_t)g.s3, (uint64_t)g.n * (uint64_t)g.n};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint64_t pl = A[i].lo * S[i];
    uint64_t ph = __umul64hi(A[i].lo, S[i]);
    // A_hi < 2^32; A_hi S 2^64 stays below 2^96 only for S < 2^32 (then no wrap)
    ok &= A[i].hi == 0 || (S[i] >> 32) == 0;
    ph += (uint64_t)(uint32_t)A[i].hi * (uint32_t)S[i];
    ok &= ph < (1ull << 32);  // product below 2^96: the sum of five stays below 2^99
    lo += pl;
    hi += ph + (lo < pl ? 1ull : 0ull);
  }
  if (!ok || hi == 0 || hi >= (1ull << 32)) return false;
  uint64_t m;
  int ex2;
  *T = round96((uint32_t)lo, (uint32_t)(lo >> 32), (uint32_t)hi, f.E, m, ex2);
  return true;
}

// Eq. 1 in single precision (the fp32 variant): coefficients rounded to float,
// the sums converted, four fused multiply-adds.
__device__ __forceinline__ float eq1_f32(const double *k, const BatchAgg &g) {
  if (g.n == 0) return 0.0f;
  float T = __double2float_rn(k[0]);
  T = __fmaf_rn(__double2float_rn(k[1]), (float)g.s1, T);
  T = __fmaf_rn(__double2float_rn(k[2]), (float)g.s2, T);
  T = __fmaf_rn(__double2float_rn(k[3]), (float)g.s3, T);
  T = __fmaf_rn(__double2float_rn(k[4]), (float)(g.n * g.n), T);
  return T;
}

// Single-precision share coefficients of a segment and batch size n:
// {K = fl(beta/n) + fl(a4 n), a1, a2, a3}.
struct Share32 {
  float K, a1, a2, a3;
};

__device__ __forceinline__ Share32 share32_const(const double *k, int64_t n) {
  const float fn = (float)n;
  Share32 r;
  r.K = n > 0 ? __fadd_rn(__fdiv_rn(__double2float_rn(k[0]), fn), __fmul_rn(__double2float_rn(k[4]), fn)) : 0.0f;
  r.a1 = __double2float_rn(k[1]);
  r.a2 = __double2float_rn(k[2]);
  r.a3 = __double2float_rn(k[3]);
  return r;
}

// K + p (a1 + a3 p) + a2 c in fused multiply-adds.
__device__ __forceinline__ float share_f32(const Share32 &q, int32_t p, int32_t c) {
  const float fp = (float)p;
  return __fmaf_rn(q.a2, (float)c, __fmaf_rn(__fmaf_rn(q.a3, fp, q.a1), fp, q.K));
}

// Per-batch share constant: q = fl(beta/n), a4n = fl(a4*n), kf = fix(fl(q+a4n)).
__device__ __forceinline__ KEntry batch_k(const ModelP &mp, int s, int64_t n, bool *slow) {
  if (n >= 1 && n <= mp.nk) {
    const KEntry e = mp.ktab[s * (mp.nk + 1) + n];
    if (mp.fixed && e.kf.hi == kKSlowHi) *slow = true;
    return e;
  }
  KEntry e;
  const double *k = mp.coef[s];
  const double dn = (double)n;
  e.q = __ddiv_rn(k[0], dn);
  e.a4n = __dmul_rn(k[4], dn);
  e.kf = mk128(0, 0);
  if (mp.fixed) {
    bool ovf = false;
    e.kf = double_to_fix(__dadd_rn(e.q, e.a4n), mp.fx[s].E, &ovf);
    if (ovf) *slow = true;
  }
  return e;
}

__device__ __forceinline__ double share_fp64(const double *k, double q, double a4n, int64_t p, int64_t c) {
  double t = q;
  t = __dadd_rn(t, __dmul_rn(k[1], (double)p));
  t = __dadd_rn(t, __dmul_rn(k[2], (double)c));
  t = __dadd_rn(t, __dmul_rn(k[3], (double)(p * p)));
  t = __dadd_rn(t, a4n);
  return t;
}

// 0 <= a < 2^64 times 0 <= x < 2^32, exact (at most 96 bits).
__device__ __forceinline__ i128 mul_u64_u32(uint64_t a, uint32_t x) {
  const uint64_t lo = (uint64_t)(uint32_t)a * x;
  const uint64_t hi = (a >> 32) * (uint64_t)x;
  i128 r;
  r.lo = lo + (hi << 32);
  r.hi = (hi >> 32) + (r.lo < lo ? 1ull : 0ull);
  return r;
}

__device__ __forceinline__ i128 a2_times(const SegFix &f, uint32_t c) {
  return f.a2_narrow ? mul_u64_u32(f.A2.lo, c) : mul128_u32(f.A2, c);
}

// share = kf + (A1 + A3 p) p + A2 c, exact, then one rounding.  0 <= p <= 2^24.
template <class F>
__device__ __forceinline__ Rounded share_fix(const F &f, i128 kf, uint32_t p, uint32_t c) {
  i128 V;
  if (p == 1) {
    V = add128(kf, f.A13);
  } else {
    const i128 r = add128(f.A1, mul128_u32(f.A3, p));
    V = add128(kf, mul128_u32(r, p));
  }
  V = add128(V, f.a2_narrow ? mul_u64_u32(f.A2.lo, c) : mul128_u32(f.A2, c));
  return fix_to_double_pos(V, f.E);
}

__device__ __forceinline__ Rounded decompose(double d) {
  Rounded r;
  const uint64_t b = (uint64_t)__double_as_longlong(d);
  r.d = d;
  r.neg = (b >> 63) != 0;
  const int be = (int)((b >> 52) & 0x7FF);
  r.m = b & ((1ull << 52) - 1);
  if (be == 0) {
    r.ex = -1074;
  } else {
    r.m |= 1ull << 52;
    r.ex = be - 1075;
  }
  if (r.m == 0) r.neg = false;
  return r;
}

// ---------------------------------------------------------------- tenant accumulation
//
// Every share is rounded to a multiple of 2^-72 s (exact for shares of at least
// 2^-20 s) and added EXACTLY into per-tenant 128-bit integers.  Integer addition
// is associative, so the totals are the same whatever the order of the
// additions: deterministic without ordering the reduction.  Within a CTA the
// hot tenants (ids < H) live in shared memory as four 32-bit words with exact
// carry propagation through the atomics' return values; the CTA adds its
// table into global per-tenant words at the end, and ids >= H go there
// directly.  The global words hold 32-bit limbs in 64-bit counters and are
// folded into the exact state by k_tenant_fold.

__device__ __forceinline__ i128 share_to_tenant_fix(const Rounded &r, int *bad) {
  const int sh = r.ex - kTenLsb;
  if (!r.neg && sh >= 0 && sh <= 10) return mk128(r.m << sh, 0);  // common case: fits 64 bits
  if (r.m == 0) return mk128(0, 0);
  i128 q;
  if (sh >= 0) {
    if (sh > 127 - 54) {
      *bad = 1;
      return mk128(0, 0);
    }
    q = shl128(r.m, 0, sh);
  } else {
    const int rs = -sh;
    if (rs > 60) return mk128(0, 0);
    uint64_t v = r.m >> rs;
    const uint64_t rem = r.m & ((1ull << rs) - 1);
    const uint64_t half = 1ull << (rs - 1);
    if (rem > half || (rem == half && (v & 1ull))) ++v;
    q = mk128(v, 0);
  }
  return r.neg ? neg128(q) : q;
}

// Global pending words of tenant u: four 32-bit limbs (top one signed), each
// accumulated in a 64-bit counter.
__device__ __forceinline__ void pend_add(unsigned long long *pend, int64_t u, i128 q) {
  unsigned long long *w = pend + 4 * u;
  const unsigned long long l0 = q.lo & 0xffffffffull, l1 = q.lo >> 32, l2 = q.hi & 0xffffffffull;
  const long long l3 = (long long)q.hi >> 32;
  if (l0) atomicAdd(w + 0, l0);
  if (l1) atomicAdd(w + 1, l1);
  if (l2) atomicAdd(w + 2, l2);
  if (l3) atomicAdd(w + 3, (unsigned long long)l3);
}

// Shared-memory tenant table.  Each hot tenant has kTenRep replicas of a
// 128-bit integer held as four 32-bit words; a thread adds into replica
// (threadIdx.x & (kTenRep - 1)).  Word k of replica r of tenant u is
// tt[k * plane + r * stride + u]: consecutive tenants fall in consecutive
// banks and, the stride being 8 mod 32 words, one tenant's replicas would fall
// in different banks.  One replica measured fastest on the Zipf workloads (more
// divide same-tenant conflicts but cost shared memory and flush work).
constexpr int kTenRep = 1;
__host__ __device__ constexpr int ten_stride(int H) { return ((H + 31) & ~31) + 8; }
__host__ __device__ constexpr int ten_plane(int H) { return kTenRep * ten_stride(H); }
__host__ __device__ constexpr size_t ten_bytes(int H) { return 4 * sizeof(uint32_t) * (size_t)ten_plane(H); }

// Word 0 of this thread's replica of tenant u (word k is k * ten_plane(H) further).
__device__ __forceinline__ uint32_t *ten_word0(uint32_t *tt, int H, int u) {
  return tt + (threadIdx.x & (kTenRep - 1)) * ten_stride(H) + u;
}

// Exact q into the 128-bit integer whose word k is w[k * plane].  Each word's
// atomic returns its old value, so the thread whose addition wraps a word is
// the one that carries into the next: the multi-word sum stays exact (mod
// 2^128) under any interleaving.
__device__ __forceinline__ void hot_add(uint32_t *w, int plane, i128 q) {
  const uint32_t v[4] = {(uint32_t)q.lo, (uint32_t)(q.lo >> 32), (uint32_t)q.hi, (uint32_t)(q.hi >> 32)};
  uint32_t c = 0;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint32_t add = v[k] + c;
    uint32_t cc = (add < v[k]) ? 1u : 0u;
    if (add) {
      const uint32_t o = atomicAdd(w + k * plane, add);
      cc |= (o + add < o) ? 1u : 0u;
    }
    c = cc;
  }
}

// Tenant u's total over the replicas (mod 2^128).
__device__ __forceinline__ i128 hot_value(const uint32_t *tt, int H, int u) {
  const int S = ten_stride(H), P = ten_plane(H);
  i128 v = mk128(0, 0);
#pragma unroll
  for (int r = 0; r < kTenRep; ++r) {
    const uint32_t *w = tt + r * S + u;
    v = add128(v, mk128((uint64_t)w[0] | ((uint64_t)w[P] << 32), (uint64_t)w[2 * P] | ((uint64_t)w[3 * P] << 32)));
  }
  return v;
}

// ---------------------------------------------------------------- per-batch and per-request steps

enum : int {
  M_ATTR = 1,    // T (if a.T) and shares (if a.share)
  M_TEN = 4,     // accumulate tenant totals (with M_ATTR)
  M_FEAT = 8,    // write batch features / segment codes only
  M_FIX = 16,    // fixed-point arithmetic (else fp64)
  M_FIT = 32,    // accumulate the least-squares statistics (with M_FEAT's reduction)
  M_F32 = 64,    // single-precision T and shares (into a.T32 / a.share32), with M_ATTR
};

// Per-segment integers the share path needs, kept in shared memory so that a
// runtime segment index is one shared-memory load (not a select over kernel
// parameters).
struct SegS {
  i128 A1, A3, A13, A2;
  int E;
  int a2_narrow;
  int p_narrow;  // 1: 0 <= A1 < 2^95 and 0 <= A3 < 2^64 (prefill constant in 128 bits)
  int pad;
};

// fx: the segments' fixed-point parameters (a shared-memory copy in k_warps,
// where the lanes of a warp take different segments).
template <int MODE>
__device__ __forceinline__ void emit_batch(const TileArgs &a, int64_t gb, const BatchAgg &g, int s, const SegFix *fx) {
  if (MODE & M_FEAT) {
    if (a.bfeat) {
      a.bfeat[gb] = g.s1;
      a.bfeat[a.n_batch + gb] = g.s2;
      a.bfeat[2 * a.n_batch + gb] = g.s3;
      a.bfeat[3 * a.n_batch + gb] = g.n;
      a.bfeat[4 * a.n_batch + gb] = g.n * g.n;
    }
    if (a.bseg) a.bseg[gb] = (uint8_t)s;
  }
  if ((MODE & M_ATTR) && (MODE & M_F32) && a.T32) a.T32[gb] = eq1_f32(a.mp.coef[s], g);
  if ((MODE & M_ATTR) && !(MODE & M_F32) && a.T) {
    double T;
    if (!(MODE & M_FIX))
      T = eq1_fp64(a.mp.coef[s], g);
    else if (!eq1_fast(fx[s], g, &T))
      T = eq1_fix(a.mp, s, g);
    a.T[gb] = T;
  }
}

__device__ __forceinline__ void check_req(int32_t &p, int32_t &c, int32_t &ph, int *bad) {
  if (p < 0) { p = 0; *bad = 1; }
  if (c < 0) { c = 0; *bad = 1; }
  if (ph != 0 && ph != 1) { ph = ph != 0; *bad = 1; }
}

__device__ __forceinline__ void tenant_add(const TileArgs &a, uint32_t *tt, int32_t u, const Rounded &r, int *bad) {
  if (u < 0 || u >= a.n_tenants) {
    *bad = 1;
    u = u < 0 ? 0 : a.n_tenants - 1;
  }
  const i128 q = share_to_tenant_fix(r, bad);
  if ((q.lo | q.hi) == 0) return;
  if (u < a.H)
    hot_add(ten_word0(tt, a.H, u), ten_plane(a.H), q);
  else
    pend_add(a.ten_pend, u, q);
}

// Out-of-line fp64 share (fp64 mode, very large p, or a batch constant outside
// the fixed-point range).
__device__ __noinline__ Rounded share_slow(const ModelP &mp, int s, bool fixed, i128 kf, int32_t p, int32_t c,
                                           int64_t n) {
  double q, a4n;
  if (fixed) {
    bool dummy = false;
    const KEntry e = batch_k(mp, s, n, &dummy);
    q = e.q;
    a4n = e.a4n;
  } else {
    q = __longlong_as_double((long long)kf.lo);
    a4n = __longlong_as_double((long long)kf.hi);
  }
  return decompose(share_fp64(mp.coef[s], q, a4n, p, c));
}

// ---------------------------------------------------------------- tenant pass 2

// state[u] += pending limbs of u; pending limbs cleared.  Deterministic: pure
// integer arithmetic on exact sums.
__global__ void k_tenant_fold(unsigned long long *__restrict__ pend, i128 *__restrict__ state, int32_t n_tenants,
                              int *status) {
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= n_tenants) return;
  unsigned long long *w = pend + 4 * (int64_t)u;
  const long long w0 = (long long)w[0], w1 = (long long)w[1], w2 = (long long)w[2], w3 = (long long)w[3];
  if ((w0 | w1 | w2 | w3) == 0) return;
  i128 v = mk128((uint64_t)w0, (uint64_t)(w0 >> 63));
  v = add128(v, shl128((uint64_t)w1, (uint64_t)(w1 >> 63), 32));
  v = add128(v, mk128(0, (uint64_t)w2));
  v = add128(v, mk128(0, (uint64_t)w3 << 32));
  const i128 old = state[u];
  const i128 nw = add128(old, v);
  // overflow of the signed 128-bit total (|total| >= 2^127 * 2^-72 s = 2^55 s)
  if (is_neg128(old) == is_neg128(v) && is_neg128(nw) != is_neg128(old)) flag(status, kStatusData);
  state[u] = nw;
  w[0] = w[1] = w[2] = w[3] = 0;
}

__global__ void k_tenant_totals(const i128 *__restrict__ state, double *__restrict__ L, int32_t n_tenants) {
  const int u = blockIdx.x * blockDim.x + threadIdx.x;
  if (u >= n_tenants) return;
  L[u] = fix_to_double(state[u], kTenLsb).d;
}

// Standalone pass 1 over given shares: grid-stride, hot tenants in shared memory.
__global__ void __launch_bounds__(kBlock) k_tenant_acc(const double *__restrict__ share,
                                                        const int32_t *__restrict__ ten, int64_t n,
                                                        unsigned long long *pend, int32_t n_tenants, int32_t H,
                                                        int *status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  uint32_t *tt = reinterpret_cast<uint32_t *>(smem_raw);
  for (int i = threadIdx.x; i < 4 * ten_plane(H); i += kBlock) tt[i] = 0;
  __syncthreads();
  int bad = 0;
  TileArgs a{};
  a.n_tenants = n_tenants;
  a.H = H;
  a.ten_pend = pend;
  const int64_t stride = (int64_t)gridDim.x * kBlock;
  for (int64_t i = blockIdx.x * (int64_t)kBlock + threadIdx.x; i < n; i += stride) {
    tenant_add(a, tt, __ldcs(ten + i), decompose(__ldcs(share + i)), &bad);
  }
  if (bad) flag(status, kStatusData);
  __syncthreads();
  for (int u = threadIdx.x; u < H; u += kBlock) {
    const i128 v = hot_value(tt, H, u);
    if (v.lo | v.hi) pend_add(pend, u, v);
  }
}

// ---------------------------------------------------------------- small kernels

// K table: for every segment and 1 <= n <= nk, q = fl(beta/n), a4n = fl(a4*n),
// kf = fl(q + a4n) at the segment's fixed-point scale.
__global__ void k_ktable(ModelP mp, KEntry *tab) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  const int per = mp.nk + 1;
  if (idx >= 4 * per) return;
  const int s = idx / per, n = idx % per;
  KEntry e;
  if (n == 0) {
    e.q = 0;
    e.a4n = 0;
    e.kf = mk128(0, 0);
  } else {
    const double *k = mp.coef[s];
    e.q = __ddiv_rn(k[0], (double)n);
    e.a4n = __dmul_rn(k[4], (double)n);
    bool ovf = false;
    e.kf = mp.fixed ? double_to_fix(__dadd_rn(e.q, e.a4n), mp.fx[s].E, &ovf) : mk128(0, 0);
    if (ovf) e.kf = mk128(0, kKSlowHi);
  }
  tab[idx] = e;
}

// Signed 64-bit product with overflow detection.
__device__ __forceinline__ bool mul_ovf(int64_t x, int64_t y, long long *r) {
  const long long lo = (long long)((uint64_t)x * (uint64_t)y);
  const long long hi = __mul64hi((long long)x, (long long)y);
  *r = lo;
  return hi != (lo >> 63);
}

// Physical per-request features p*phi0, c*phi1, p^2*phi2 (int64, SoA [3][n]).
__global__ void k_req_features(const int32_t *__restrict__ p, const int32_t *__restrict__ c, int64_t n,
                               int64_t phi0, int64_t phi1, int64_t phi2, int64_t *__restrict__ out, int *status) {
  int bad = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t pi = p[i], ci = c[i];
    long long v0, v1, v2;
    const bool o0 = mul_ovf(pi, phi0, &v0);
    const bool o1 = mul_ovf(ci, phi1, &v1);
    const bool o2 = mul_ovf(pi * pi, phi2, &v2);
    if (o0 || o1 || o2 || pi < 0 || ci < 0) bad = 1;
    __stcs((long long *)out + i, o0 ? INT64_MAX : v0);
    __stcs((long long *)out + n + i, o1 ? INT64_MAX : v1);
    __stcs((long long *)out + 2 * n + i, o2 ? INT64_MAX : v2);
  }
  if (bad) flag(status, kStatusData);
}

// Eq. 1 from precomputed aggregates.
template <bool FIX>
__global__ void k_batch_latency(ModelP mp, const int64_t *__restrict__ feat, const uint8_t *__restrict__ seg,
                                int64_t nb, double *__restrict__ T, int *status) {
  int bad = 0;
  for (int64_t b = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; b < nb; b += (int64_t)gridDim.x * blockDim.x) {
    BatchAgg g{feat[b], feat[nb + b], feat[2 * nb + b], feat[3 * nb + b], 0};
    int s = seg[b];
    if (s > 3) {
      bad = 1;
      s &= 3;
    }
    if (g.s1 < 0 || g.s2 < 0 || g.s3 < 0 || g.n < 0) {
      bad = 1;
      T[b] = 0.0;
      continue;
    }
    T[b] = FIX ? eq1_fix(mp, s, g) : eq1_fp64(mp.coef[s], g);
  }
  if (bad) flag(status, kStatusData);
}

}  // namespace lv
