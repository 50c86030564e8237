// Device code for the LLMVisor attribution path (sm_103a).
//
// Tiling.  The work is a merge of two sorted streams: batch boundaries
// (offsets) and requests.  Batch b starts at merge position f(b) = b + off[b]
// (b boundaries and off[b] requests precede it); f is strictly increasing, so
// cutting the merge sequence every kD positions gives tiles that each own the
// batches whose start falls inside them -- at most kD batches and about kD
// requests, whatever the batch-size distribution (merge-based partitioning,
// Merrill & Garland, SC'16).  A tile holds whole batches and needs no data from
// its neighbours.  The partition is written by one coalesced pass over the
// offsets (k_partition); no search is needed.
//
// Pipeline.  k_tiles runs persistent CTAs (two per SM).  Each CTA walks its
// tiles with a two-stage ring in shared memory: while the threads compute tile
// k, bulk asynchronous copies (TMA) bring the offsets window and the request
// arrays of tile k+1.  Per tile, every thread takes K consecutive requests, the
// per-batch sums S1 = sum p, S2 = sum c, S3 = sum p^2 and the prefill count
// come from a block-wide prefix sum sampled at batch boundaries (exact integer
// sums), then each batch's segment, T and per-request constant are computed
// once and every request's share is produced from registers.  A batch with
// more requests than the staging capacity takes a block-wide path that reads
// global memory directly.
#pragma once

#include <cstddef>
#include <cstdint>

#include "lv_fixed.cuh"
#include "lv_tma.cuh"

namespace lv {

constexpr int kBlock = 256;                        // threads per CTA
constexpr int kD = 1024;                           // merge positions per tile (batches + requests)
constexpr int kCap = 1280;                         // requests staged per tile
constexpr int kK = (kCap + kBlock - 1) / kBlock;   // max requests per thread per sub-tile
constexpr int kBPT = kD / kBlock;                  // max batches per thread in the per-batch phase
constexpr int kHotMax = 512;                       // tenants kept in shared memory per CTA
constexpr int kNK = 256;                           // per-batch constants cached in shared memory for n <= kNK
constexpr int64_t kPMaxFix = 1ll << 24;            // p beyond this uses the fp64 share path
constexpr int kTenLsb = -72;                       // tenant totals: shares rounded to 2^-72 s, summed exactly

constexpr int kStatusData = 1;
constexpr int kStatusTimeout = 2;
constexpr int kStatusOverflow = 4;

struct SegFix {
  i128 A1, A2, A3;   // exact a_k * 2^-E
  i128 B, A4;        // beta and a4 at 2^E (rounded to nearest)
  i128 A13;          // A1 + A3: the p-terms of a decode request (p = 1)
  uint64_t lim[4];   // exact T path valid when S1, S2, S3, n^2 <= lim[0..3]
  int E;
  int a2_narrow;     // 1: 0 <= A2 < 2^64 (64-bit multiply suffices)
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
  double *T, *share;
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

// ---------------------------------------------------------------- block scan

struct Sums {
  int64_t s1, s2, s3;
  int32_t ph;
};

__device__ __forceinline__ Sums warp_incl_scan(Sums v, int lane) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int64_t a = __shfl_up_sync(0xffffffffu, v.s1, d);
    const int64_t b = __shfl_up_sync(0xffffffffu, v.s2, d);
    const int64_t c = __shfl_up_sync(0xffffffffu, v.s3, d);
    const int32_t e = __shfl_up_sync(0xffffffffu, v.ph, d);
    if (lane >= d) {
      v.s1 += a;
      v.s2 += b;
      v.s3 += c;
      v.ph += e;
    }
  }
  return v;
}

// Exclusive block scan; `scr` holds kBlock/32 Sums.  Contains __syncthreads.
__device__ __forceinline__ Sums block_excl_scan(Sums v, Sums *scr) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  Sums inc = warp_incl_scan(v, lane);
  if (lane == 31) scr[wid] = inc;
  __syncthreads();
  if (wid == 0) {
    Sums w = lane < kBlock / 32 ? scr[lane] : Sums{0, 0, 0, 0};
    Sums wi = warp_incl_scan(w, lane);
    if (lane < kBlock / 32) {
      Sums ex{wi.s1 - w.s1, wi.s2 - w.s2, wi.s3 - w.s3, wi.ph - w.ph};
      scr[lane] = ex;
    }
  }
  __syncthreads();
  Sums base = scr[wid];
  Sums r{base.s1 + inc.s1 - v.s1, base.s2 + inc.s2 - v.s2, base.s3 + inc.s3 - v.s3, base.ph + inc.ph - v.ph};
  __syncthreads();
  return r;
}

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
// exact range.
__device__ __forceinline__ double eq1_fix(const ModelP &mp, int s, const BatchAgg &g) {
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

// Exact q into the 128-bit integer held as four 32-bit shared-memory words.
// Each word's atomic returns its old value, so the thread whose addition
// wraps a word is the one that carries into the next: the multi-word sum stays
// exact (mod 2^128) under any interleaving.
__device__ __forceinline__ void hot_add(uint32_t *w, i128 q) {
  if (q.hi == 0) {
    const uint32_t lo = (uint32_t)q.lo, hi = (uint32_t)(q.lo >> 32);
    uint32_t c = 0;
    if (lo) {
      const uint32_t o = atomicAdd(w, lo);
      c = (o + lo < o) ? 1u : 0u;
    }
    const uint32_t add1 = hi + c;
    uint32_t c1 = (add1 < hi) ? 1u : 0u;
    if (add1) {
      const uint32_t o = atomicAdd(w + 1, add1);
      c1 |= (o + add1 < o) ? 1u : 0u;
    }
    if (c1) {
      const uint32_t o = atomicAdd(w + 2, 1u);
      if (o == 0xffffffffu) atomicAdd(w + 3, 1u);
    }
    return;
  }
  const uint32_t v[4] = {(uint32_t)q.lo, (uint32_t)(q.lo >> 32), (uint32_t)q.hi, (uint32_t)(q.hi >> 32)};
  uint32_t c = 0;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint32_t add = v[k] + c;
    uint32_t cc = (add < v[k]) ? 1u : 0u;
    if (add) {
      const uint32_t o = atomicAdd(w + k, add);
      cc |= (o + add < o) ? 1u : 0u;
    }
    c = cc;
  }
}

__device__ __forceinline__ i128 hot_value(const uint32_t *w) {
  return mk128((uint64_t)w[0] | ((uint64_t)w[1] << 32), (uint64_t)w[2] | ((uint64_t)w[3] << 32));
}

// ---------------------------------------------------------------- the tile kernel

enum : int {
  M_ATTR = 1,    // T (if a.T) and shares (if a.share)
  M_TEN = 4,     // accumulate tenant totals (with M_ATTR)
  M_FEAT = 8,    // write batch features / segment codes only
  M_FIX = 16,    // fixed-point arithmetic (else fp64)
  M_FIT = 32,    // accumulate the least-squares statistics (with M_FEAT's reduction)
};

// One stage of the ring: offsets window and request arrays of one tile.
struct Stage {
  alignas(16) int64_t win[kD + 4];
  alignas(16) int32_t sp[kCap + 8];
  alignas(16) int32_t sc[kCap + 8];
  alignas(16) int32_t sph[kCap + 8];
  alignas(16) int32_t sten[kCap + 8];
};

struct TileHdr {
  int64_t b0, b1, r0, r1, staged, lo;
};

// Per-segment integers the share path needs, kept in shared memory so that a
// runtime segment index is one shared-memory load (not a select over kernel
// parameters).
struct SegS {
  i128 A1, A3, A13, A2;
  int E;
  int a2_narrow;
  int pad[2];
};

struct Smem {
  Stage st[2];
  union U {
    struct {
      alignas(16) int64_t s1[kD + 4];
      alignas(16) int64_t s2[kD + 4];
      alignas(16) int64_t s3[kD + 4];
      alignas(16) int32_t ph[kD + 4];
    } pre;
    struct {
      alignas(16) i128 kf[kD];  // per-batch constant (fixed) or {q, a4n} (fp64)
      alignas(16) uint8_t seg[kD];
    } bp;
  } u;
  alignas(16) double kcd[4][kNK + 1];  // fl(fl(beta/n) + fl(a4*n)) for n <= kNK
  alignas(16) uint8_t fseg[kD + 16];   // fit mode: segment of each batch of the sub-tile
  alignas(16) SegS seg[4];
  TileHdr hdr[2];
  alignas(16) Sums scr[kBlock / 32];
  alignas(8) uint64_t full[2];
  int flags;
};
static_assert(offsetof(Stage, win) % 16 == 0 && offsetof(Stage, sp) % 16 == 0 && offsetof(Stage, sc) % 16 == 0 &&
                  offsetof(Stage, sph) % 16 == 0 && offsetof(Stage, sten) % 16 == 0 && sizeof(Stage) % 16 == 0,
              "bulk-copy destinations must be 16-byte aligned");
static_assert(offsetof(Stage, sc) - offsetof(Stage, sp) == sizeof(int32_t) * (kCap + 8) &&
                  2 * sizeof(int32_t) * (kCap + 8) >= sizeof(double) * kCap,
              "shares are staged over the consumed p and c arrays");
static_assert(sizeof(Smem) % 16 == 0, "tenant table follows Smem");

// Loads tile t's extent from the partition (clamped: never trusted blindly).
__device__ __forceinline__ TileHdr tile_info(const TileArgs &a, int64_t t, int *bad) {
  const TilePart p0 = a.part[t], p1 = a.part[t + 1];
  TileHdr h;
  h.b0 = clampi(p0.b, 0, a.n_batch);
  h.b1 = clampi(p1.b, h.b0, a.n_batch);
  if (h.b1 - h.b0 > kD) {
    h.b1 = h.b0 + kD;
    *bad = 1;
  }
  h.r0 = clampi(p0.r, 0, a.n_req);
  h.r1 = clampi(p1.r, h.r0, a.n_req);
  h.staged = h.r1 - h.r0 < kCap ? h.r1 - h.r0 : kCap;
  h.lo = h.b0 & ~1ll;
  return h;
}

// Thread 0: fill stage `s` with the tile described by h (window by bulk copy,
// request arrays by bulk copy, ragged ends by plain loads), then arrive on the
// stage's barrier with the byte count.
template <bool TEN>
__device__ __forceinline__ void issue_tile(const TileArgs &a, Smem &sm, int s, const TileHdr &h) {
  Stage &st = sm.st[s];
  uint64_t *bar = &sm.full[s];
  sm.hdr[s] = h;
  // window [lo, hi): 16-byte aligned start, even element count, never past off[n_batch]
  const int64_t w_up = (h.b1 + 2) & ~1ll, w_cap = (a.n_batch + 1) & ~1ll;
  const int64_t hi_w = w_up < w_cap ? w_up : w_cap;
  if (hi_w <= h.b1) st.win[h.b1 - h.lo] = h.r1;  // last boundary not covered by the copy
  // requests [base, vend) by bulk copy; [max(vend, base), r0 + staged) by plain loads
  const int64_t base = h.r0 & ~3ll;
  const int64_t rend = h.r0 + h.staged;
  const int64_t vup = (rend + 3) & ~3ll, vcap = a.n_req & ~3ll;
  const int64_t vend = vup < vcap ? vup : vcap;
  for (int64_t g = (vend > base ? vend : base); g < rend; ++g) {
    const int i = (int)(g - base);
    st.sp[i] = a.p[g];
    st.sc[i] = a.c[g];
    st.sph[i] = a.ph[g];
    if (TEN) st.sten[i] = a.ten[g];
  }
  const uint32_t wbytes = hi_w > h.lo ? (uint32_t)(hi_w - h.lo) * 8u : 0u;
  const uint32_t rbytes = vend > base ? (uint32_t)(vend - base) * 4u : 0u;
  const uint32_t bytes = wbytes + rbytes * (TEN ? 4u : 3u);
  mbar_arrive_expect_tx(bar, bytes);
  if (wbytes) bulk_g2s(st.win, a.off + h.lo, wbytes, bar);
  if (rbytes) {
    bulk_g2s(st.sp, a.p + base, rbytes, bar);
    bulk_g2s(st.sc, a.c + base, rbytes, bar);
    bulk_g2s(st.sph, a.ph + base, rbytes, bar);
    if (TEN) bulk_g2s(st.sten, a.ten + base, rbytes, bar);
  }
}

template <int MODE>
__device__ __forceinline__ void emit_batch(const TileArgs &a, int64_t gb, const BatchAgg &g, int s) {
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
  if ((MODE & M_ATTR) && a.T) {
    a.T[gb] = (MODE & M_FIX) ? eq1_fix(a.mp, s, g) : eq1_fp64(a.mp.coef[s], g);
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
    hot_add(tt + 4 * u, q);
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

// Share of one request (kf: per-batch constant; in fp64 mode kf holds {q, a4n}).
template <int MODE>
__device__ __forceinline__ Rounded one_share(const TileArgs &a, const SegS *segs, int s, bool slow, i128 kf,
                                             int32_t p, int32_t c, int64_t n) {
  if ((MODE & M_FIX) && !slow && p <= kPMaxFix) return share_fix(segs[s], kf, (uint32_t)p, (uint32_t)c);
  return share_slow(a.mp, s, (MODE & M_FIX) != 0, kf, p, c, n);
}

// Per-batch constant for the share phase, as stored in Smem::bp.
template <int MODE>
__device__ __forceinline__ i128 batch_const(const TileArgs &a, const Smem &sm, int s, int64_t n, bool *slow) {
  if (MODE & M_FIX) {
    if (n >= 1 && n <= kNK) {
      bool ovf = false;
      const i128 kf = double_to_fix(sm.kcd[s][n], sm.seg[s].E, &ovf);
      if (ovf) *slow = true;
      return kf;
    }
    return batch_k(a.mp, s, n, slow).kf;
  }
  bool dummy = false;
  const KEntry e = batch_k(a.mp, s, n, &dummy);
  return mk128((uint64_t)__double_as_longlong(e.q), (uint64_t)__double_as_longlong(e.a4n));
}

// Block-wide path for one batch with more than kCap requests (reads global memory).
template <int MODE>
__device__ void jumbo_batch(const TileArgs &a, Smem &sm, uint32_t *tt, int64_t gb, int64_t r0, int64_t r1,
                            FitAcc &facc, int *bad) {
  Sums acc{0, 0, 0, 0};
  for (int64_t i = r0 + threadIdx.x; i < r1; i += kBlock) {
    int32_t p = a.p[i], c = a.c[i], ph = a.ph[i];
    check_req(p, c, ph, bad);
    acc.s1 += p;
    acc.s2 += c;
    acc.s3 += (int64_t)p * p;
    acc.ph += ph;
  }
  const Sums ex = block_excl_scan(acc, sm.scr);
  if (threadIdx.x == kBlock - 1) sm.scr[0] = Sums{ex.s1 + acc.s1, ex.s2 + acc.s2, ex.s3 + acc.s3, ex.ph + acc.ph};
  __syncthreads();
  const Sums tot = sm.scr[0];
  __syncthreads();
  const BatchAgg g{tot.s1, tot.s2, tot.s3, r1 - r0, tot.ph > 0};
  const int s = segment_of(a.mp, g);
  if (threadIdx.x == 0) emit_batch<MODE>(a, gb, g, s);
  if (MODE & M_FIT) {
    const int NE = fit_entries(a.fit.n_y);
    const int64_t x[5] = {1, g.s1, g.s2, g.s3, g.n * g.n};
    const bool in_range = g.s1 < kFitFeatMax && g.s2 < kFitFeatMax && g.s3 < kFitFeatMax && x[4] < kFitFeatMax;
    if (!in_range && threadIdx.x == 0) flag(a.status, kStatusOverflow);
    if ((int)threadIdx.x < 4 * NE && (int)threadIdx.x / NE == s && in_range)
      fit_owner_add(facc, threadIdx.x % NE, a.fit.n_y, x, a.fit.y, a.n_batch, gb, g.s1 != g.s3, bad);
  }
  if (MODE & M_ATTR) {
    bool slow = false;
    const i128 kf = batch_const<MODE>(a, sm, s, g.n, &slow);
    for (int64_t i = r0 + threadIdx.x; i < r1; i += kBlock) {
      int32_t p = a.p[i], c = a.c[i], ph = a.ph[i];
      int dummy = 0;
      check_req(p, c, ph, &dummy);
      const Rounded r = one_share<MODE>(a, sm.seg, s, slow, kf, p, c, g.n);
      if (a.share) __stcs(a.share + i, r.d);
      if (MODE & M_TEN) tenant_add(a, tt, a.ten[i], r, bad);
    }
  }
}

// Requests [r0, win[nbt]) of whole batches 0..nbt-1 of `win` (global batch
// index gb0 + j), staged in `st` from element `base`.
template <int MODE>
__device__ __forceinline__ void sub_tile(const TileArgs &a, Smem &sm, Stage &st, uint32_t *tt, const int64_t *win,
                                         int64_t gb0, int nbt, int64_t r0, int64_t base, FitAcc &facc, int *bad) {
  constexpr bool kTen = (MODE & M_TEN) != 0;
  constexpr bool kShares = (MODE & M_ATTR) != 0;
  const int tid = threadIdx.x;
  const int64_t r1 = win[nbt];
  const int nr = (int)(r1 - r0);
  const int o = (int)(r0 - base);

  // ---- per-thread requests [i0, i1)
  const int K = (nr + kBlock - 1) / kBlock;
  const int i0 = min(tid * K, nr), i1 = min(i0 + K, nr);
  const int t_last = nr > 0 ? (nr - 1) / K : 0;
  int jf;  // first boundary j with q_j >= i0
  {
    int l = 0, h = nbt + 1;
    while (l < h) {
      const int m = (l + h) >> 1;
      if (win[m] - r0 < i0) l = m + 1; else h = m;
    }
    jf = l;
  }
  Sums acc{0, 0, 0, 0};
  int j = jf;
  int32_t rp[kK], rc[kK], rt[kK];
#pragma unroll
  for (int k = 0; k < kK; ++k) {
    const int i = i0 + k;
    if (k < K && i < i1) {
      while (j <= nbt && win[j] - r0 == i) {
        sm.u.pre.s1[j] = acc.s1;
        sm.u.pre.s2[j] = acc.s2;
        sm.u.pre.s3[j] = acc.s3;
        sm.u.pre.ph[j] = acc.ph;
        ++j;
      }
      int32_t p = st.sp[o + i], c = st.sc[o + i], ph = st.sph[o + i];
      check_req(p, c, ph, bad);
      rp[k] = p;
      rc[k] = c;
      if (kTen) rt[k] = st.sten[o + i];
      acc.s1 += p;
      acc.s2 += c;
      acc.s3 += (int64_t)p * p;
      acc.ph += ph;
    }
  }
  if (tid == t_last) {
    while (j <= nbt && win[j] - r0 == nr) {
      sm.u.pre.s1[j] = acc.s1;
      sm.u.pre.s2[j] = acc.s2;
      sm.u.pre.s3[j] = acc.s3;
      sm.u.pre.ph[j] = acc.ph;
      ++j;
    }
  }
  const int jend = j;
  const Sums base_s = block_excl_scan(acc, sm.scr);
  for (int jj = jf; jj < jend; ++jj) {
    sm.u.pre.s1[jj] += base_s.s1;
    sm.u.pre.s2[jj] += base_s.s2;
    sm.u.pre.s3[jj] += base_s.s3;
    sm.u.pre.ph[jj] += base_s.ph;
  }
  __syncthreads();

  // ---- per batch: aggregates, segment, outputs, share constant
  int segv[kBPT];
  i128 kv[kBPT];
  bool slowv[kBPT];
#pragma unroll
  for (int m = 0; m < kBPT; ++m) {
    const int jb = tid + m * kBlock;
    if (jb < nbt) {
      BatchAgg g;
      g.s1 = sm.u.pre.s1[jb + 1] - sm.u.pre.s1[jb];
      g.s2 = sm.u.pre.s2[jb + 1] - sm.u.pre.s2[jb];
      g.s3 = sm.u.pre.s3[jb + 1] - sm.u.pre.s3[jb];
      g.n = win[jb + 1] - win[jb];
      g.prefill = (sm.u.pre.ph[jb + 1] - sm.u.pre.ph[jb]) > 0;
      const int s = segment_of(a.mp, g);
      segv[m] = s;
      emit_batch<MODE>(a, gb0 + jb, g, s);
      if (MODE & M_FIT) {
        const bool in_range = g.s1 < kFitFeatMax && g.s2 < kFitFeatMax && g.s3 < kFitFeatMax &&
                              g.n * g.n < kFitFeatMax;
        if (!in_range) flag(a.status, kStatusOverflow);
        sm.fseg[jb] = (g.n > 0 && in_range) ? (uint8_t)s : (uint8_t)0xff;
      }
      slowv[m] = false;
      kv[m] = mk128(0, 0);
      if (kShares && g.n > 0) kv[m] = batch_const<MODE>(a, sm, s, g.n, &slowv[m]);
    }
  }
  if (!kShares) {
    __syncthreads();
    if (MODE & M_FIT) {
      // owners: thread (g, e) adds the batches of group g of this sub-tile
      const int NE = fit_entries(a.fit.n_y);
      if (tid < 4 * NE) {
        const int g = tid / NE, e = tid % NE;
        for (int jb = 0; jb < nbt; ++jb) {
          if (sm.fseg[jb] != g) continue;
          const int64_t n = win[jb + 1] - win[jb];
          const int64_t x[5] = {1, sm.u.pre.s1[jb + 1] - sm.u.pre.s1[jb], sm.u.pre.s2[jb + 1] - sm.u.pre.s2[jb],
                                sm.u.pre.s3[jb + 1] - sm.u.pre.s3[jb], n * n};
          fit_owner_add(facc, e, a.fit.n_y, x, a.fit.y, a.n_batch, gb0 + jb, x[1] != x[3], bad);
        }
      }
      __syncthreads();
    }
    return;
  }
  __syncthreads();  // pre[] is dead from here on; bp[] aliases it
#pragma unroll
  for (int m = 0; m < kBPT; ++m) {
    const int jb = tid + m * kBlock;
    if (jb < nbt) {
      sm.u.bp.kf[jb] = kv[m];
      sm.u.bp.seg[jb] = (uint8_t)(segv[m] | (slowv[m] ? 0x80 : 0));
    }
  }
  __syncthreads();

  // ---- shares from registers; staged over the consumed p/c arrays
  double *shs = reinterpret_cast<double *>(st.sp);
  int jb = jf > 0 ? jf - 1 : 0;  // batch of request i0: last j with q_j <= i0
  while (jb + 1 <= nbt && win[jb + 1] - r0 <= i0) ++jb;
#pragma unroll
  for (int k = 0; k < kK; ++k) {
    const int i = i0 + k;
    if (k < K && i < i1) {
      while (win[jb + 1] - r0 <= i) ++jb;
      const uint8_t sg = sm.u.bp.seg[jb];
      const Rounded r = one_share<MODE>(a, sm.seg, sg & 3, (sg & 0x80) != 0, sm.u.bp.kf[jb], rp[k], rc[k],
                                        win[jb + 1] - win[jb]);
      shs[i] = r.d;
      if (kTen) tenant_add(a, tt, rt[k], r, bad);
    }
  }
  __syncthreads();
  if (a.share) {
    for (int i = tid; i < nr; i += kBlock) __stcs(a.share + r0 + i, shs[i]);
  }
  __syncthreads();
}

template <int MODE>
__global__ void __launch_bounds__(kBlock, 2) k_tiles(const TileArgs a) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Smem &sm = *reinterpret_cast<Smem *>(smem_raw);
  uint32_t *tt = reinterpret_cast<uint32_t *>(smem_raw + sizeof(Smem));
  const int tid = threadIdx.x;
  constexpr bool kTen = (MODE & M_TEN) != 0;
  int bad = 0;
  FitAcc facc;
  facc.w[0] = facc.w[1] = facc.w[2] = facc.w[3] = 0;

  if (kTen) {
    for (int i = tid; i < 4 * a.H; i += kBlock) tt[i] = 0;
  }
  if ((MODE & M_FIX) && (MODE & M_ATTR)) {
    for (int i = tid; i < 4 * (kNK + 1); i += kBlock) {
      const int s = i / (kNK + 1), n = i % (kNK + 1);
      double v = 0.0;
      if (n >= 1 && n <= a.mp.nk) {
        const KEntry e = a.mp.ktab[s * (a.mp.nk + 1) + n];
        v = __dadd_rn(e.q, e.a4n);
      }
      sm.kcd[s][n] = v;
    }
    if (tid < 4) {
      const SegFix &f = a.mp.fx[tid];
      SegS g;
      g.A1 = f.A1;
      g.A3 = f.A3;
      g.A13 = f.A13;
      g.A2 = f.A2;
      g.E = f.E;
      g.a2_narrow = f.a2_narrow;
      g.pad[0] = g.pad[1] = 0;
      sm.seg[tid] = g;
    }
  }
  if (tid == 0) {
    mbar_init(&sm.full[0], 1);
    mbar_init(&sm.full[1], 1);
    fence_mbar_init();
  }
  __syncthreads();

  const int64_t G = gridDim.x;
  TileHdr nxt{};
  if (tid == 0 && (int64_t)blockIdx.x < a.n_tiles) {
    const TileHdr h0 = tile_info(a, blockIdx.x, &bad);
    issue_tile<kTen>(a, sm, 0, h0);
    if ((int64_t)blockIdx.x + G < a.n_tiles) nxt = tile_info(a, blockIdx.x + G, &bad);
  }

  int64_t k = 0;
  for (int64_t t = blockIdx.x; t < a.n_tiles; t += G, ++k) {
    const int s = (int)(k & 1);
    if (tid == 0 && t + G < a.n_tiles) {
      fence_proxy_async_smem();  // the other stage was read and written by generic accesses
      issue_tile<kTen>(a, sm, s ^ 1, nxt);
      if (t + 2 * G < a.n_tiles) nxt = tile_info(a, t + 2 * G, &bad);
    }
    const bool ok = mbar_wait_bounded(&sm.full[s], (uint32_t)((k >> 1) & 1));
    if (__syncthreads_or(!ok)) {
      if (tid == 0) {
        flag(a.status, kStatusTimeout);
        // let the other stage's copies land before the CTA leaves
        if (t + G < a.n_tiles) mbar_wait_bounded(&sm.full[s ^ 1], (uint32_t)(((k + 1) >> 1) & 1));
      }
      __syncthreads();
      return;
    }
    Stage &st = sm.st[s];
    const TileHdr h = sm.hdr[s];
    const int nb = (int)(h.b1 - h.b0);
    int64_t *win = st.win + (h.b0 - h.lo);
    if (nb > 0) {
      // clamp the window into the tile's request range and check it is monotone
      for (int i = tid; i <= nb; i += kBlock) win[i] = clampi(win[i], h.r0, h.r1);
      __syncthreads();
      int nonmono = (tid == 0) && (win[0] != h.r0 || win[nb] != h.r1);
      for (int i = tid; i < nb; i += kBlock) nonmono |= win[i + 1] < win[i];
      if (__syncthreads_or(nonmono)) {
        if (tid == 0) {
          win[0] = h.r0;
          for (int i = 1; i <= nb; ++i)
            if (win[i] < win[i - 1]) win[i] = win[i - 1];
          win[nb] = h.r1;
        }
        bad = 1;
        __syncthreads();
      }
      int bs = 0;
      while (bs < nb) {
        const int64_t r0s = win[bs];
        int lo = bs, hi = nb;  // largest be in (bs, nb] with win[be] - r0s <= kCap
        if (win[nb] - r0s <= kCap) lo = nb;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (win[mid] - r0s <= kCap) lo = mid; else hi = mid - 1;
        }
        const int be = lo;
        if (be == bs) {
          jumbo_batch<MODE>(a, sm, tt, h.b0 + bs, r0s, win[bs + 1], facc, &bad);
          __syncthreads();
          bs = be + 1;
          continue;
        }
        int64_t base = h.r0 & ~3ll;
        if (bs > 0) {
          // beyond the bulk-copied range: stage this sub-tile with plain loads
          base = r0s & ~3ll;
          const int64_t r1s = win[be];
          for (int64_t g = base + tid; g < r1s; g += kBlock) {
            const int i = (int)(g - base);
            st.sp[i] = a.p[g];
            st.sc[i] = a.c[g];
            st.sph[i] = a.ph[g];
            if (kTen) st.sten[i] = a.ten[g];
          }
          __syncthreads();
        }
        sub_tile<MODE>(a, sm, st, tt, win + bs, h.b0 + bs, be - bs, r0s, base, facc, &bad);
        bs = be;
      }
    }
    __syncthreads();  // stage s is free for the next issue
  }
  if (bad) flag(a.status, kStatusData);
  if (MODE & M_FIT) {
    const int NE = fit_entries(a.fit.n_y);
    if (tid < 4 * NE) a.fit.partial[(int64_t)blockIdx.x * 4 * NE + tid] = facc;
  }
  if (kTen) {
    __syncthreads();
    for (int u = tid; u < a.H; u += kBlock) {
      const i128 v = hot_value(tt + 4 * u);
      if (v.lo | v.hi) pend_add(a.ten_pend, u, v);
    }
  }
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
  for (int i = threadIdx.x; i < 4 * H; i += kBlock) tt[i] = 0;
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
    const i128 v = hot_value(tt + 4 * u);
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
