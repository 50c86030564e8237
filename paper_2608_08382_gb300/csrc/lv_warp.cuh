// Warp-centric attribution kernels (sm_103a).
//
// Every step of the path is a stream over request arrays, so the kernels are
// built to keep many independent warps busy with coalesced loads and no
// block-wide barrier while tiles are processed.
//
// Work decomposition.  The merge of batch boundaries and requests is cut every
// kDW positions (k_partition); a warp tile owns the batches whose start falls
// in its window (whole batches, no data shared with neighbours).  Persistent
// warps take tiles from a global counter and walk each tile 32 batches at a
// time, batch b0 + j on lane j:
//   - a batch of kBig..kJumbo requests is reduced by the whole warp with
//     coalesced strided loads and a butterfly sum; its segment and per-request
//     constant follow (uniform across the warp) and its shares come from a
//     second strided pass while its requests are still in L1;
//   - batches of fewer than kBig requests are packed into rounds of up to 32
//     requests (whole batches per round, one request per lane), reduced with a
//     segmented scan across lanes and attributed in a second sweep of the same
//     rounds;
//   - a batch of more than kJumbo requests is queued for k_jumbo, where a whole
//     CTA takes it, so that no warp holds a disproportionate share of the work;
//   - T, the batch features and the fit statistics of the 32 batches are then
//     produced with one lane per batch.
// All sums are exact integers, so results do not depend on this schedule.
#pragma once

#include <cooperative_groups.h>

#include "lv_kernels.cuh"

namespace lv {

constexpr int kWarps = 16;                 // warps per CTA of k_warps
constexpr int kWThreads = 32 * kWarps;
constexpr int kDW = 1024;                  // merge positions per warp tile (large inputs: 2 kDW)
constexpr int kJumbo = 512;                // larger batches are attributed by k_jumbo
constexpr int kBig = 32;                   // batches with at least this many requests are processed warp-strided
constexpr int kJBlock = 512;               // threads per CTA of k_jumbo
constexpr int kJWarps = kJBlock / 32;
constexpr unsigned kFull = 0xffffffffu;

static_assert(kJumbo <= kNK * 4, "jumbo threshold");

// Shared memory of k_warps; the tenant table (4 x H words) and, in fit mode,
// the per-warp fit accumulators ([kWarps][4 * NE]) follow it.
struct WSmem {
  alignas(16) i128 kfix[4][kNK + 1];     // K at 2^E for n <= kNK (fixed-point mode)
  alignas(16) SegS seg[4];
  alignas(16) uint8_t kslow[4][kNK + 4];  // 1: K outside the fixed-point range
  alignas(16) uint8_t owner[kWarps][32];  // small-batch rounds: head slot -> lane
  alignas(16) Sums gsum[kWarps][32];      // sums of the group's big batches (kept out of registers)
  alignas(16) SegFix fx[4];               // Eq. 1 parameters (lanes of a warp read different segments)
};
static_assert(sizeof(WSmem) % 16 == 0, "tenant table follows WSmem");

// Shared memory of k_jumbo (tenant table follows).
struct JSmem {
  alignas(16) SegS seg[4];
  alignas(16) Sums red[kJWarps];
  alignas(16) Sums tot;
};
static_assert(sizeof(JSmem) % 16 == 0, "tenant table follows JSmem");

__device__ __forceinline__ Sums add_sums(Sums a, const Sums &b) {
  a.s1 += b.s1;
  a.s2 += b.s2;
  a.s3 += b.s3;
  a.ph += b.ph;
  return a;
}

__device__ __forceinline__ Sums shfl_sums(const Sums &v, int src) {
  return Sums{__shfl_sync(kFull, v.s1, src), __shfl_sync(kFull, v.s2, src), __shfl_sync(kFull, v.s3, src),
              __shfl_sync(kFull, v.ph, src)};
}

__device__ __forceinline__ Sums warp_sum(Sums v) {
#pragma unroll
  for (int d = 16; d; d >>= 1) {
    v.s1 += __shfl_xor_sync(kFull, v.s1, d);
    v.s2 += __shfl_xor_sync(kFull, v.s2, d);
    v.s3 += __shfl_xor_sync(kFull, v.s3, d);
    v.ph += __shfl_xor_sync(kFull, v.ph, d);
  }
  return v;
}

// Warp sum of per-lane sums over at most 16 requests each (s1, s2 below 2^35,
// ph at most 16; s3 modulo 2^64, as 64-bit adds take it), from 32-bit warp
// reductions of 27-bit pieces: 32 of them sum below 2^32.
__device__ __forceinline__ Sums warp_sum16(const Sums &v) {
  constexpr uint32_t kM27 = (1u << 27) - 1u;
  const uint64_t a = (uint64_t)v.s1, b = (uint64_t)v.s2, c = (uint64_t)v.s3;
  const uint32_t a0 = __reduce_add_sync(kFull, (uint32_t)a & kM27), a1 = __reduce_add_sync(kFull, (uint32_t)(a >> 27));
  const uint32_t b0 = __reduce_add_sync(kFull, (uint32_t)b & kM27), b1 = __reduce_add_sync(kFull, (uint32_t)(b >> 27));
  const uint32_t c0 = __reduce_add_sync(kFull, (uint32_t)c & kM27);
  const uint32_t c1 = __reduce_add_sync(kFull, (uint32_t)(c >> 27) & kM27);
  const uint32_t c2 = __reduce_add_sync(kFull, (uint32_t)(c >> 54));
  Sums r;
  r.s1 = (int64_t)(((uint64_t)a1 << 27) + a0);
  r.s2 = (int64_t)(((uint64_t)b1 << 27) + b0);
  r.s3 = (int64_t)(((uint64_t)c2 << 54) + ((uint64_t)c1 << 27) + c0);
  r.ph = (int32_t)__reduce_add_sync(kFull, (uint32_t)v.ph);
  return r;
}

__device__ __forceinline__ int warp_excl_scan_int(int v, int lane) {
  int x = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int y = __shfl_up_sync(kFull, x, d);
    if (lane >= d) x += y;
  }
  return x - v;
}

__device__ __forceinline__ void prefetch_l2(const void *p) { asm volatile("prefetch.global.L2 [%0];" ::"l"(p)); }

// ---------------------------------------------------------------- decode fast path
//
// A decode request (p = 1) of a batch with constant K has the exact share
// V = K13 + A2 c with K13 = K + A1 + A3.  When A2 < 2^64 (the segment's
// a2_narrow) this is one 64x32-bit product and a 128-bit add; the result is
// rounded to double with 32-bit funnel shifts.  Requests the fast loops do not
// cover (p != 1, V outside [2^64, 2^96), a tenant contribution outside the
// three-word range) are left to defer_one, 32 at a time: it takes the same
// steps with K + p (A1 + A3 p) in place of K13 (prefill_const) where that is
// exact, and the general path, exact for every case, otherwise.

// v = k + (a1:a0) * c, four 32-bit words, exact (the sum stays below 2^128):
// carry-propagating multiply-adds, low word first.
__device__ __forceinline__ void mad_k13(uint32_t k0, uint32_t k1, uint32_t k2, uint32_t k3, uint32_t a0, uint32_t a1,
                                        uint32_t c, uint32_t &v0, uint32_t &v1, uint32_t &v2, uint32_t &v3) {
  asm("mad.lo.cc.u32 %0, %4, %6, %7;\n\t"
      "madc.hi.cc.u32 %1, %4, %6, %8;\n\t"
      "addc.cc.u32 %2, %9, 0;\n\t"
      "addc.u32 %3, %10, 0;\n\t"
      "mad.lo.cc.u32 %1, %5, %6, %1;\n\t"
      "madc.hi.cc.u32 %2, %5, %6, %2;\n\t"
      "addc.u32 %3, %3, 0;"
      : "=r"(v0), "=r"(v1), "=r"(v2), "=r"(v3)
      : "r"(a0), "r"(a1), "r"(c), "r"(k0), "r"(k1), "r"(k2), "r"(k3));
}

// Constant part of a prefill request's share, kf + p (A1 + A3 p), for a
// segment with p_narrow and p <= 2^24: A1 + A3 p < 2^96 and its product with p
// stays below 2^120, so the 128-bit sum is exact whenever the share itself is
// below 2^128 (which the caller's V < 2^96 test then confirms).
__device__ __forceinline__ void prefill_const(const SegS &sg, i128 kf, uint32_t p, uint32_t &b0, uint32_t &b1,
                                              uint32_t &b2, uint32_t &b3) {
  const i128 r = add128(sg.A1, mul_u64_u32(sg.A3.lo, p));
  const i128 b = add128(kf, mul128_u32(r, p));
  b0 = (uint32_t)b.lo;
  b1 = (uint32_t)(b.lo >> 32);
  b2 = (uint32_t)b.hi;
  b3 = (uint32_t)(b.hi >> 32);
}

// Tenant contribution of a share m * 2^ex2 (m <= 2^53) when q = m 2^(ex2+72)
// has at most three 32-bit words and the tenant id is valid; false otherwise
// (nothing is added then).  Hot tenants: exact multi-word add in shared memory;
// cold tenants: 32-bit limbs into the global 64-bit pending counters.
__device__ __forceinline__ bool tenant_fast(const TileArgs &a, uint32_t *tt, int32_t u, uint64_t m, int ex2) {
  const int sh = ex2 - kTenLsb;
  if ((unsigned)sh <= 10u && (unsigned)u < (unsigned)a.H) {
    // the common case: q = m 2^sh <= 2^63, two words
    const uint32_t ml = (uint32_t)m, mh = (uint32_t)(m >> 32);
    uint32_t *w = ten_word0(tt, a.H, u);
    const int P = ten_plane(a.H);
    const uint32_t lo = ml << sh, hi = __funnelshift_l(ml, mh, sh);
    const uint32_t o0 = atomicAdd(w, lo);
    const uint32_t a1 = hi + ((o0 + lo < o0) ? 1u : 0u);  // hi <= 2^31: no wrap
    const uint32_t o1 = atomicAdd(w + P, a1);
    if (o1 + a1 < o1) {
      if (atomicAdd(w + 2 * P, 1u) == 0xffffffffu) atomicAdd(w + 3 * P, 1u);
    }
    return true;
  }
  if ((unsigned)sh > 42u || (unsigned)u >= (unsigned)a.n_tenants) return false;
  const uint32_t ml = (uint32_t)m, mh = (uint32_t)(m >> 32);
  const bool lowp = sh < 32;
  const int t = lowp ? sh : sh - 32;
  const uint32_t x0 = ml << t, x1 = __funnelshift_l(ml, mh, t), x2 = t ? mh >> (32 - t) : 0u;
  const uint32_t q0 = lowp ? x0 : 0u, q1 = lowp ? x1 : x0, q2 = lowp ? x2 : x1;
  if (u < a.H) {
    uint32_t *w = ten_word0(tt, a.H, u);
    const int P = ten_plane(a.H);
    const uint32_t o0 = atomicAdd(w, q0);
    const uint32_t a1 = q1 + ((o0 + q0 < o0) ? 1u : 0u);
    const uint32_t o1 = atomicAdd(w + P, a1);
    const uint32_t a2 = q2 + (((o1 + a1 < o1) || a1 < q1) ? 1u : 0u);  // q2 < 2^22: no wrap
    if (a2) {
      if (atomicAdd(w + 2 * P, a2) + a2 < a2) atomicAdd(w + 3 * P, 1u);
    }
  } else {
    unsigned long long *pw = a.ten_pend + 4 * (int64_t)u;
    atomicAdd(pw, (unsigned long long)q0);
    atomicAdd(pw + 1, (unsigned long long)q1);
    if (q2) atomicAdd(pw + 2, (unsigned long long)q2);
  }
  return true;
}

// Tenant contribution of an fp32 share (the fp32 variant): its exact value
// m24 * 2^(e - 150) re-expressed with a 53-bit significand for tenant_fast;
// zero adds nothing, the rest (negative, subnormal, out of range) the general
// add of its exact double.
__device__ __forceinline__ void tenant_f32(const TileArgs &a, uint32_t *tt, int32_t u, float s, int *bad) {
  const uint32_t bits = __float_as_uint(s);
  const uint32_t e = (bits >> 23) & 0xffu;
  if (!(bits >> 31) && e != 0u && e != 0xffu) {
    const uint64_t m = (uint64_t)((bits & 0x7fffffu) | 0x800000u) << 29;
    if (tenant_fast(a, tt, u, m, (int)e - 150 - 29)) return;
  }
  if (s != 0.0f) tenant_add(a, tt, u, decompose((double)s), bad);
}

// Warp-strided fp32 shares of requests [r0, r1) of one batch (the fp32 variant:
// every request inline, no deferral).
template <int MODE>
__device__ __forceinline__ void big_shares_f32(const TileArgs &a, uint32_t *tt, const Share32 &q, int64_t r0,
                                               int64_t r1, int lane, int *bad) {
  const int32_t *P = a.p + r0, *C = a.c + r0, *U = a.ten + r0;
  float *S = a.share32 ? a.share32 + r0 : nullptr;
  const int n = (int)(r1 - r0);
  for (int q0 = lane; q0 < n; q0 += 32) {
    int32_t p = P[q0], c = C[q0];
    p = p < 0 ? 0 : p;
    c = c < 0 ? 0 : c;
    const float s = share_f32(q, p, c);
    if (S) __stcs(S + q0, s);
    if (MODE & M_TEN) tenant_f32(a, tt, U[q0], s, bad);
  }
}

// One request's share, its store and its tenant contribution.
template <int MODE>
__device__ __forceinline__ void attribute_one(const TileArgs &a, uint32_t *tt, const SegS &sg, int s, bool slow,
                                              i128 kf, int64_t n, int64_t i, int32_t p, int32_t c, int32_t u,
                                              int *bad) {
  Rounded r;
  if ((MODE & M_FIX) && !slow && p <= kPMaxFix)
    r = share_fix(sg, kf, (uint32_t)p, (uint32_t)c);
  else
    r = share_slow(a.mp, s, (MODE & M_FIX) != 0, kf, p, c, n);
  if (a.share) __stcs(a.share + i, r.d);
  if (MODE & M_TEN) tenant_add(a, tt, u, r, bad);
}

// Per-request constant of a batch: fixed-point K (from the shared table for
// n <= kNK), or {fl(beta/n), fl(a4 n)} in fp64 mode.
template <int MODE>
__device__ __forceinline__ i128 batch_const_w(const TileArgs &a, const WSmem *ws, int s, int64_t n, bool *slow) {
  if (MODE & M_FIX) {
    if (ws && n >= 1 && n <= kNK) {
      if (ws->kslow[s][n]) *slow = true;
      return ws->kfix[s][n];
    }
    return batch_k(a.mp, s, n, slow).kf;
  }
  bool dummy = false;
  const KEntry e = batch_k(a.mp, s, n, &dummy);
  return mk128((uint64_t)__double_as_longlong(e.q), (uint64_t)__double_as_longlong(e.a4n));
}

// The general path for one request (segment s, constant kf, fields p, c, u as
// loaded): the exact fixed-point share with prefill_const where the segment
// allows it, else the exact or fp64 share and the general tenant add.  Out of
// line: the fast loops send it only the requests they do not cover.
template <int MODE>
__device__ __forceinline__ void defer_one(const TileArgs &a, uint32_t *tt, const SegS *segs, int s, bool slow, i128 kf,
                                          int64_t n, int64_t q, int32_t p, int32_t c, int32_t u, int *bad) {
  p = p < 0 ? 0 : p;
  c = c < 0 ? 0 : c;
  const SegS &sg = segs[s];
  if ((MODE & M_FIX) && !slow && sg.a2_narrow && sg.p_narrow && p <= kPMaxFix) {
    uint32_t b0, b1, b2, b3, v0, v1, v2, v3;
    prefill_const(sg, kf, (uint32_t)p, b0, b1, b2, b3);
    mad_k13(b0, b1, b2, b3, (uint32_t)sg.A2.lo, (uint32_t)(sg.A2.lo >> 32), (uint32_t)c, v0, v1, v2, v3);
    if (v3 == 0u && v2 != 0u) {
      uint64_t m;
      int ex2;
      const double d = round96(v0, v1, v2, sg.E, m, ex2);
      if (!(MODE & M_TEN) || tenant_fast(a, tt, u, m, ex2)) {
        if (a.share) __stcs(a.share + q, d);
        return;
      }
    }
  }
  attribute_one<MODE>(a, tt, sg, s, slow, kf, n, q, p, c, u, bad);
}

// Requests left to the general path, gathered per warp across batches so that
// they are attributed 32 at a time with every lane busy (a batch of a
// decode-dominated workload has only a few).  meta = n << 4 | segment (other
// bits ignored); p, c, u: the request's fields as loaded (unclamped).
constexpr int kDeferCap = 64;
struct DeferList {
  int64_t q[kDeferCap];
  int meta[kDeferCap];
  int32_t p[kDeferCap], c[kDeferCap], u[kDeferCap];
};

// Attribute the first min(cnt, 32) entries, one per lane (the batch constant
// looked up again), move the rest (at most 31 when cnt < kDeferCap) to the
// front and return their number.  Out of line: once per 32 deferred requests;
// bad data is flagged in the status word directly.
template <int MODE>
__device__ __noinline__ int defer_flush(const TileArgs &a, uint32_t *tt, const WSmem &ws, DeferList &L, int cnt,
                                        int lane) {
  const int take = cnt < 32 ? cnt : 32;
  if (lane < take) {
    const int m = L.meta[lane];
    const int s = m & 3;
    const int64_t n = m >> 4;
    bool slow = false;
    int bad = 0;
    const i128 kf = batch_const_w<MODE>(a, &ws, s, n, &slow);
    defer_one<MODE>(a, tt, ws.seg, s, slow, kf, n, L.q[lane], L.p[lane], L.c[lane], L.u[lane], &bad);
    if (bad) flag(a.status, kStatusData);
  }
  const int rest = cnt - take;
  int64_t q = 0;
  int m = 0, p = 0, c = 0, u = 0;
  __syncwarp();
  if (lane < rest) {
    q = L.q[take + lane];
    m = L.meta[take + lane];
    p = L.p[take + lane];
    c = L.c[take + lane];
    u = L.u[take + lane];
  }
  __syncwarp();
  if (lane < rest) {
    L.q[lane] = q;
    L.meta[lane] = m;
    L.p[lane] = p;
    L.c[lane] = c;
    L.u[lane] = u;
  }
  __syncwarp();
  return rest;
}

// Append the request of every lane with `flag` (all lanes call); attribute 32
// at once when the list holds that many.
template <int MODE>
__device__ __forceinline__ void defer_push(const TileArgs &a, uint32_t *tt, const WSmem &ws, DeferList &L, int &cnt,
                                           bool flag, int64_t q, int meta, int32_t p, int32_t c, int32_t u, int lane) {
  const uint32_t bm = __ballot_sync(kFull, flag);
  if (!bm) return;
  if (flag) {
    const int slot = cnt + __popc(bm & ((1u << lane) - 1u));
    L.q[slot] = q;
    L.meta[slot] = meta;
    L.p[slot] = p;
    L.c[slot] = c;
    L.u[slot] = u;
  }
  cnt += __popc(bm);
  __syncwarp();
  if (cnt >= 32) cnt = defer_flush<MODE>(a, tt, ws, L, cnt, lane);
}

// Warp-strided sums over requests [r0, r1) (at most kJumbo); uniform result on
// every lane.  Indices are 32-bit offsets from the batch's first request.  With
// a tenant pass the tenant ids are loaded (and checked) here as well, so that
// the share pass finds the whole batch in L1.
__device__ __forceinline__ Sums big_reduce(const TileArgs &a, int64_t r0, int64_t r1, int lane, int *bad) {
  const int32_t *P = a.p + r0, *C = a.c + r0, *PH = a.ph + r0;
  const int n = (int)(r1 - r0);
  Sums acc{0, 0, 0, 0};
  int32_t sgn = 0, phx = 0;  // sign bits of p and c; bits of phase beyond 0/1
  for (int i = lane; i < n; i += 4 * 32) {
    int32_t p[4], c[4], ph[4], u[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      const int q = i + 32 * t;
      const bool in = q < n;
      u[t] = (in && a.ten) ? a.ten[r0 + q] : 0;
      p[t] = in ? P[q] : 0;
      c[t] = in ? C[q] : 0;
      ph[t] = in ? PH[q] : 0;
    }
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      sgn |= p[t] | c[t];
      if (a.ten && (unsigned)u[t] >= (unsigned)a.n_tenants) sgn |= 0x80000000;
      phx |= ph[t] & ~1;
      const int32_t pt = p[t] < 0 ? 0 : p[t], ct = c[t] < 0 ? 0 : c[t];
      acc.s1 += pt;
      acc.s2 += ct;
      acc.s3 += (int64_t)pt * pt;
      acc.ph += ph[t] != 0;
    }
  }
  if (sgn < 0 || phx != 0) *bad = 1;  // clamped as check_req does
  static_assert(kJumbo <= 4 * 4 * 32, "at most 16 requests per lane");
  return warp_sum16(acc);
}

// Warp-strided shares of requests [r0, r1) of one batch (segment s, constant kf):
// the general loop for fp64 mode, an out-of-range constant or a wide A2 (out
// of line: the fast loop serves the common case).
template <int MODE>
__device__ __noinline__ void big_shares(const TileArgs &a, uint32_t *tt, const SegS &sg, int s, bool slow,
                                           i128 kf, int64_t r0, int64_t r1, int lane) {
  const int64_t n = r1 - r0;
  int bad = 0;
  for (int64_t i = r0 + lane; i < r1; i += 4 * 32) {
    int32_t p[4], c[4], u[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t q = i + 32 * k;
      const bool in = q < r1;
      p[k] = in ? a.p[q] : 0;
      c[k] = in ? a.c[q] : 0;
      u[k] = (in && (MODE & M_TEN)) ? a.ten[q] : 0;
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int64_t q = i + 32 * k;
      if (q < r1) {
        const int32_t pk = p[k] < 0 ? 0 : p[k], ck = c[k] < 0 ? 0 : c[k];
        attribute_one<MODE>(a, tt, sg, s, slow, kf, n, q, pk, ck, u[k], &bad);
      }
    }
  }
  if (bad) flag(a.status, kStatusData);
}

// Warp-strided shares of a batch whose requests take the fast path
// (fixed-point mode, in-range constant kf, A2 < 2^64).  The batch was just
// reduced, tenant ids included, so its requests are in L1 and the loop takes
// one request per lane per step; every lane runs every step, so the requests
// the fast path does not cover go to the defer list as they appear.  ALLDEC:
// every p = 1, p is not loaded.
template <int MODE, bool ALLDEC>
__device__ __forceinline__ void big_shares_fast(const TileArgs &a, uint32_t *tt, const WSmem &ws, DeferList &L,
                                                int &cnt, int s, i128 kf, int64_t r0, int64_t r1, int lane) {
  const SegS &sg = ws.seg[s];
  const i128 K13 = add128(kf, sg.A13);
  const uint32_t k0 = (uint32_t)K13.lo, k1 = (uint32_t)(K13.lo >> 32), k2 = (uint32_t)K13.hi,
                 k3 = (uint32_t)(K13.hi >> 32);
  const uint32_t a0 = (uint32_t)sg.A2.lo, a1 = (uint32_t)(sg.A2.lo >> 32);
  const int E = sg.E;
  const int32_t *P = a.p + r0, *C = a.c + r0, *U = a.ten + r0;
  double *S = a.share ? a.share + r0 : nullptr;
  const int n = (int)(r1 - r0);
  const int meta = (n << 4) | s;
  for (int q0 = 0; q0 < n; q0 += 32) {
    const int q = q0 + lane;
    bool done = true;
    int32_t c0 = 0, u0 = 0, p0 = 1;
    if (q < n) {
      c0 = C[q];
      u0 = (MODE & M_TEN) ? U[q] : 0;
      p0 = ALLDEC ? 1 : P[q];
      uint32_t v0, v1, v2, v3;
      mad_k13(k0, k1, k2, k3, a0, a1, (uint32_t)(c0 < 0 ? 0 : c0), v0, v1, v2, v3);
      uint64_t m;
      int ex2;
      const double d = round96(v0, v1, v2, E, m, ex2);
      done = (ALLDEC || p0 == 1) && v3 == 0u && v2 != 0u;
      if (MODE & M_TEN) {
        if (done) done = tenant_fast(a, tt, u0, m, ex2);
      }
      if (done && S) __stcs(S + q, d);
    }
    defer_push<MODE>(a, tt, ws, L, cnt, !done, r0 + q, meta, p0, c0, u0, lane);
  }
}

// Rounds over the small batches of a group (lanes with `small`): every round
// takes the next batches whose requests fit in 32 slots, one request per lane.
// A segmented scan gives each batch's sums to its lane (`mys`).  With
// attribution the same round then forms those batches' constants on their
// lanes and attributes the round's requests, whose fields are still in
// registers: a batch lies within one round.  pn: the lane's request count (0
// for other lanes); P: exclusive prefix of pn; base = o0 - P so that slot q of
// the lane's batch is request base + q.  meta = n << 4 | fast << 3 | slow << 2
// | segment.
template <int MODE>
__device__ __forceinline__ void small_rounds(const TileArgs &a, const WSmem &ws, uint32_t *tt, uint8_t *owner,
                                             DeferList *dl, int &dcnt, bool small, int pn, int P, int64_t base,
                                             Sums &mys, int lane, int *bad) {
  uint32_t rem = __ballot_sync(kFull, small);
  while (rem) {
    const int start = __shfl_sync(kFull, P, __ffs(rem) - 1);
    const bool in = ((rem >> lane) & 1u) && (P + pn <= start + 32);
    const uint32_t rm = __ballot_sync(kFull, in);
    rem &= ~rm;
    if (in) owner[P - start] = (uint8_t)lane;
    const uint32_t H = __reduce_or_sync(kFull, in ? (1u << (P - start)) : 0u);
    __syncwarp();
    const int len = __shfl_sync(kFull, P + pn, 31 - __clz(rm)) - start;
    const bool act = lane < len;
    const int hp = act ? 31 - __clz(H & ((2u << lane) - 1u)) : 0;  // head slot of this lane's batch
    const int j = owner[hp];
    const int64_t r = __shfl_sync(kFull, base, j) + start + lane;
    Sums v{0, 0, 0, 0};
    int32_t p = 0, c = 0, ph = 0;
    if (act) {
      p = a.p[r];
      c = a.c[r];
      ph = a.ph[r];
      check_req(p, c, ph, bad);  // clamped: the share paths clamp the same way
      v = Sums{p, c, (int64_t)p * p, ph};
    }
    const int maxn = __reduce_max_sync(kFull, in ? pn : 0);
    for (int d = 1; d < maxn; d <<= 1) {
      const Sums w{__shfl_up_sync(kFull, v.s1, d), __shfl_up_sync(kFull, v.s2, d),
                   __shfl_up_sync(kFull, v.s3, d), __shfl_up_sync(kFull, v.ph, d)};
      if (lane - d >= hp) v = add_sums(v, w);
    }
    const Sums tot = shfl_sums(v, in ? P - start + pn - 1 : 0);
    if (in) mys = tot;
    if ((MODE & M_ATTR) && (MODE & M_F32)) {
      Share32 mq{0.0f, 0.0f, 0.0f, 0.0f};
      if (in) {
        const BatchAgg g{mys.s1, mys.s2, mys.s3, pn, mys.ph > 0};
        mq = share32_const(a.mp.coef[segment_of(a.mp, g)], pn);
      }
      const Share32 q{__shfl_sync(kFull, mq.K, j), __shfl_sync(kFull, mq.a1, j), __shfl_sync(kFull, mq.a2, j),
                      __shfl_sync(kFull, mq.a3, j)};
      if (act) {
        const float s = share_f32(q, p, c);
        if (a.share32) __stcs(a.share32 + r, s);
        if (MODE & M_TEN) tenant_f32(a, tt, a.ten[r], s, bad);
      }
    } else if (MODE & M_ATTR) {
      i128 myk = mk128(0, 0);
      int mymeta = 0;
      if (in) {
        const BatchAgg g{mys.s1, mys.s2, mys.s3, pn, mys.ph > 0};
        const int s = segment_of(a.mp, g);
        bool slow = false;
        myk = batch_const_w<MODE>(a, &ws, s, pn, &slow);
        const bool fast = (MODE & M_FIX) && !slow && ws.seg[s].a2_narrow;
        mymeta = (pn << 4) | (fast ? 8 : 0) | (slow ? 4 : 0) | s;
      }
      const uint64_t klo = __shfl_sync(kFull, myk.lo, j), khi = __shfl_sync(kFull, myk.hi, j);
      const int meta = __shfl_sync(kFull, mymeta, j);
      bool done = true;
      int32_t u = 0;
      if (act) {
        done = false;
        u = (MODE & M_TEN) ? a.ten[r] : 0;
        if (meta & 8) {
          const SegS &sg = ws.seg[meta & 3];
          const i128 K13 = add128(mk128(klo, khi), sg.A13);
          uint32_t v0, v1, v2, v3;
          mad_k13((uint32_t)K13.lo, (uint32_t)(K13.lo >> 32), (uint32_t)K13.hi, (uint32_t)(K13.hi >> 32),
                  (uint32_t)sg.A2.lo, (uint32_t)(sg.A2.lo >> 32), (uint32_t)c, v0, v1, v2, v3);
          uint64_t m;
          int ex2;
          const double d = round96(v0, v1, v2, sg.E, m, ex2);
          done = p == 1 && v3 == 0u && v2 != 0u;
          if (MODE & M_TEN) {
            if (done) done = tenant_fast(a, tt, u, m, ex2);
          }
          if (done && a.share) __stcs(a.share + r, d);
        }
      }
      defer_push<MODE>(a, tt, ws, *dl, dcnt, !done, r, meta, p, c, u, lane);
    }
    __syncwarp();  // owner[] is rewritten by the next round
  }
}

// Fit statistics of the group's batches into this warp's accumulators
// fw[group][entry].  Entry order: 15 Gram pairs (a <= b, row order), 5 X^T y
// columns per y vector, one y'y per y vector, one flag.  Every entry adds
// x[a] * B for each batch of its group, B a 192-bit two's complement operand:
// a feature (Gram), the batch's Y = y * 2^100 (X^T y), or floor(Y^2 / 2^64)
// with x[a] = 1 (y'y).  The batches of segment g are taken kFitRecs at a time:
// their owner lanes write the batches' records (kFitRecWords words: x0..x4 =
// 1, S1, S2, S3, n^2, a zero word, then Y and floor(Y^2 / 2^64), three words
// each, per y vector) to the warp's slots in shared memory, and lane e reads
// entry e's two operands from each and multiply-adds in registers, the same
// instructions for every kind of entry.  The accumulators are loaded and
// stored once per segment and group.  The record slots use the shared table
// of per-request constants, which the fit does not use.
constexpr int kFitRecWords = 6 + 6 * kFitMaxY;
constexpr int kFitRecs = 4;
static_assert(sizeof(uint64_t) * kWarps * kFitRecs * kFitRecWords <= sizeof(i128) * 4 * (kNK + 1),
              "fit record slots fit in the per-request constant table");

struct FitRole {
  int xa, b0, b1, b2;  // record words of x and of B's three words
};

__device__ __forceinline__ FitRole fit_role(int e, int n_y) {
  if (e < 15) {
    int a = 0, r = e;
    while (r >= 5 - a) {
      r -= 5 - a;
      ++a;
    }
    return FitRole{a, a + r, 5, 5};
  }
  if (e < 15 + 5 * n_y) {
    const int col = (e - 15) % 5, kk = (e - 15) / 5;
    return FitRole{col, 6 + 6 * kk, 7 + 6 * kk, 8 + 6 * kk};
  }
  if (e < 15 + 6 * n_y) {
    const int kk = e - 15 - 5 * n_y;
    return FitRole{0, 9 + 6 * kk, 10 + 6 * kk, 11 + 6 * kk};
  }
  return FitRole{1, 3, 5, 5};  // the flag (S1 != S3) and lanes past the last entry
}

// acc += x * B (mod 2^256) for B = b0 + b1 2^64 + b2 2^128, b2 sign-extended.
__device__ __forceinline__ void fit_mac(uint64_t *acc, uint64_t x, uint64_t b0, uint64_t b1, uint64_t b2) {
  const uint64_t b3 = (uint64_t)((int64_t)b2 >> 63);
  acc_add256(acc, x * b0, __umul64hi(x, b0), __umul64hi(x, b1), __umul64hi(x, b2));
  acc_add256(acc, 0, x * b1, x * b2, x * b3);
}

// One entry's update for the record in `rec`; the flag entry ORs S1 != S3.
__device__ __forceinline__ void fit_entry(uint64_t *acc, const uint64_t *rec, const FitRole &r, bool flag) {
  const uint64_t x = rec[r.xa], b0 = rec[r.b0];
  if (flag)
    acc[0] |= x != b0 ? 1ull : 0ull;
  else
    fit_mac(acc, x, b0, rec[r.b1], rec[r.b2]);
}

__device__ __forceinline__ void fit_group(const TileArgs &a, FitAcc *fw, uint64_t *rec, int64_t g0, const Sums &mys,
                                          int64_t n, int fseg, int lane, int *bad) {
  if (!__any_sync(kFull, fseg >= 0)) return;
  const int NE = fit_entries(a.fit.n_y), n_y = a.fit.n_y;
  // this lane's batch: latencies in fixed point and floor(Y^2 / 2^64)
  i128 Ym[kFitMaxY];
  uint64_t YYm[kFitMaxY][3];
#pragma unroll
  for (int q = 0; q < kFitMaxY; ++q) {
    Ym[q] = mk128(0, 0);
    YYm[q][0] = YYm[q][1] = YYm[q][2] = 0;
    if (q < n_y && fseg >= 0) {
      bool ovf = false;
      i128 Y = y_fixed(a.fit.y[q * a.n_batch + g0 + lane], &ovf);
      if (ovf) *bad = 1;
      Ym[q] = Y;
      if (is_neg128(Y)) Y = neg128(Y);
      const uint64_t l = Y.lo, h = Y.hi;
      uint64_t w[4] = {__umul64hi(l, l), h * h, __umul64hi(h, h), 0};
      acc_add256(w, h * l, __umul64hi(h, l), 0, 0);
      acc_add256(w, h * l, __umul64hi(h, l), 0, 0);
      YYm[q][0] = w[0];
      YYm[q][1] = w[1];
      YYm[q][2] = w[2];
    }
  }
  const FitRole r0 = fit_role(lane, n_y), r1 = fit_role(lane + 32, n_y);
  const bool two = NE > 32;  // lanes 0..NE-33 also own entry lane + 32
  if (lane < kFitRecs) {
    rec[lane * kFitRecWords] = 1;
    rec[lane * kFitRecWords + 5] = 0;
  }
#pragma unroll 1
  for (int g = 0; g < 4; ++g) {
    uint32_t m = __ballot_sync(kFull, fseg == g);
    if (!m) continue;
    uint64_t acc0[4] = {0, 0, 0, 0}, acc1[4] = {0, 0, 0, 0};
    FitAcc *f0 = fw + g * NE + lane, *f1 = f0 + 32;
    if (lane < NE) {
#pragma unroll
      for (int w = 0; w < 4; ++w) acc0[w] = f0->w[w];
    }
    if (two && lane + 32 < NE) {
#pragma unroll
      for (int w = 0; w < 4; ++w) acc1[w] = f1->w[w];
    }
    while (m) {
      uint32_t sel = 0;  // the next (at most) kFitRecs batches of the segment
#pragma unroll
      for (int i = 0; i < kFitRecs; ++i) {
        sel |= m & (0u - m);
        m &= m - 1;
      }
      const int cnt = __popc(sel);
      __syncwarp();  // the previous records have been read
      if ((sel >> lane) & 1u) {
        uint64_t *rw = rec + __popc(sel & ((1u << lane) - 1u)) * kFitRecWords;
        rw[1] = (uint64_t)mys.s1;
        rw[2] = (uint64_t)mys.s2;
        rw[3] = (uint64_t)mys.s3;
        rw[4] = (uint64_t)(n * n);
#pragma unroll
        for (int q = 0; q < kFitMaxY; ++q) {
          if (q < n_y) {
            rw[6 + 6 * q] = Ym[q].lo;
            rw[7 + 6 * q] = Ym[q].hi;
            rw[8 + 6 * q] = (uint64_t)((int64_t)Ym[q].hi >> 63);
            rw[9 + 6 * q] = YYm[q][0];
            rw[10 + 6 * q] = YYm[q][1];
            rw[11 + 6 * q] = YYm[q][2];
          }
        }
      }
      __syncwarp();
      for (int i = 0; i < cnt; ++i) {
        const uint64_t *rr = rec + i * kFitRecWords;
        fit_entry(acc0, rr, r0, lane == NE - 1);
        if (two) fit_entry(acc1, rr, r1, lane + 32 == NE - 1);
      }
    }
    if (lane < NE) {
#pragma unroll
      for (int w = 0; w < 4; ++w) f0->w[w] = acc0[w];
    }
    if (two && lane + 32 < NE) {
#pragma unroll
      for (int w = 0; w < 4; ++w) f1->w[w] = acc1[w];
    }
  }
  __syncwarp();  // the record slot is rewritten by the next group
}

// One group of up to 32 consecutive batches [g0, g0 + ng) of a tile.
template <int MODE>
__device__ __forceinline__ void process_group(const TileArgs &a, WSmem &ws, uint32_t *tt, uint8_t *owner,
                                              DeferList *dl, int &dcnt, FitAcc *fw, uint64_t *frec, int64_t g0, int ng,
                                              int lane, int *bad) {
  constexpr bool kAttr = (MODE & M_ATTR) != 0;
  const bool valid = lane < ng;
  int64_t o0 = valid ? a.off[g0 + lane] : 0;
  int n = 0;  // requests of this lane's batch; 0 for jumbo batches (k_jumbo's)
  bool jumbo = false;
  {
    int64_t o1 = __shfl_down_sync(kFull, o0, 1);
    if (valid && lane == ng - 1) o1 = a.off[g0 + lane + 1];
    if (valid) {
      const int64_t c0 = clampi(o0, 0, a.n_req), c1 = clampi(o1, c0, a.n_req);
      if (c0 != o0 || c1 != o1) *bad = 1;
      o0 = c0;
      jumbo = c1 - c0 > kJumbo;
      n = jumbo ? 0 : (int)(c1 - c0);
    }
  }
  if (jumbo) {
    const unsigned long long slot = atomicAdd(a.jumbo_n, 1ull);
    if (slot < (unsigned long long)a.jumbo_cap)
      a.jumbo[slot] = g0 + lane;
    else
      *bad = 1;
  }
  Sums mys{0, 0, 0, 0};
  Sums *gsum = ws.gsum[threadIdx.x >> 5];

  // ---- big batches: reduce, constant and shares one batch at a time
  const uint32_t big0 = __ballot_sync(kFull, n >= kBig);
  uint32_t big = big0;
  while (big) {
    const int j = __ffs(big) - 1;
    big &= big - 1;
    const int64_t r0 = __shfl_sync(kFull, o0, j), r1 = r0 + __shfl_sync(kFull, n, j);
    {
      // the next 256 requests (the batches after this one) into L2 while this
      // batch is reduced and attributed: one line per lane, 8 per array.  Not
      // bounded by the tile: measured faster than stopping at its end.
      const int32_t *arr = lane < 8 ? a.p : lane < 16 ? a.c : lane < 24 ? a.ph : a.ten;
      const int64_t pq = (r1 & ~(int64_t)31) + 32 * (lane & 7);
      if (arr && pq < a.n_req) prefetch_l2(arr + pq);
    }
    const Sums tot = big_reduce(a, r0, r1, lane, bad);
    if (lane == j) gsum[j] = tot;
    if (kAttr && (MODE & M_F32)) {
      const BatchAgg g{tot.s1, tot.s2, tot.s3, r1 - r0, tot.ph > 0};
      const Share32 q = share32_const(a.mp.coef[segment_of(a.mp, g)], r1 - r0);
      big_shares_f32<MODE>(a, tt, q, r0, r1, lane, bad);
    } else if (kAttr) {
      const BatchAgg g{tot.s1, tot.s2, tot.s3, r1 - r0, tot.ph > 0};
      const int s = segment_of(a.mp, g);
      bool slow = false;
      const i128 kf = batch_const_w<MODE>(a, &ws, s, r1 - r0, &slow);
      if ((MODE & M_FIX) && !slow && ws.seg[s].a2_narrow) {
        if (tot.s1 == r1 - r0 && tot.s3 == r1 - r0)
          big_shares_fast<MODE, true>(a, tt, ws, *dl, dcnt, s, kf, r0, r1, lane);
        else
          big_shares_fast<MODE, false>(a, tt, ws, *dl, dcnt, s, kf, r0, r1, lane);
      } else {
        big_shares<MODE>(a, tt, ws.seg[s], s, slow, kf, r0, r1, lane);
      }
    }
  }

  if ((big0 >> lane) & 1u) mys = gsum[lane];  // slot j is written and read by lane j only

  // ---- small batches: packed rounds
  const bool small = n > 0 && n < kBig;
  if (__any_sync(kFull, small)) {
    const int pn = small ? n : 0;
    const int P = warp_excl_scan_int(pn, lane);
    const int64_t base = o0 - P;
    small_rounds<MODE>(a, ws, tt, owner, dl, dcnt, small, pn, P, base, mys, lane, bad);
  }

  // ---- per batch: T, features; fit statistics
  int fseg = -1;
  if (valid && !jumbo) {
    const BatchAgg g{mys.s1, mys.s2, mys.s3, n, mys.ph > 0};
    const int s = segment_of(a.mp, g);
    emit_batch<MODE>(a, g0 + lane, g, s, ws.fx);
    if (MODE & M_FIT) {
      const bool in_range = g.s1 < kFitFeatMax && g.s2 < kFitFeatMax && g.s3 < kFitFeatMax &&
                            (int64_t)n * n < kFitFeatMax;
      if (!in_range) flag(a.status, kStatusOverflow);
      if (n > 0 && in_range) fseg = s;
    }
  }
  if (MODE & M_FIT) fit_group(a, fw, frec, g0, mys, n, fseg, lane, bad);
}

// Shared-memory tables of a CTA: per-segment share parameters and, in
// fixed-point attribution, the per-request constants for n <= kNK.
template <int MODE>
__device__ __forceinline__ void init_segs(const TileArgs &a, SegS *seg) {
  if (threadIdx.x < 4) {
    const SegFix &f = a.mp.fx[threadIdx.x];
    SegS g;
    g.A1 = f.A1;
    g.A3 = f.A3;
    g.A13 = f.A13;
    g.A2 = f.A2;
    g.E = f.E;
    g.a2_narrow = f.a2_narrow;
    g.p_narrow = ((uint64_t)f.A1.hi < (1ull << 31) && f.A3.hi == 0) ? 1 : 0;
    g.pad = 0;
    seg[threadIdx.x] = g;
  }
}

template <int MODE>
__global__ void __launch_bounds__(kWThreads, 2) k_warps(const TileArgs a) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  WSmem &ws = *reinterpret_cast<WSmem *>(smem_raw);
  uint32_t *tt = reinterpret_cast<uint32_t *>(smem_raw + sizeof(WSmem));
  constexpr bool kTen = (MODE & M_TEN) != 0;
  constexpr bool kFit = (MODE & M_FIT) != 0;
  static_assert(!(kFit && (MODE & M_ATTR)), "fit records share the attribution constant table");
  FitAcc *facc = reinterpret_cast<FitAcc *>(smem_raw + sizeof(WSmem) + (kTen ? ten_bytes(a.H) : 0));
  DeferList *dlists = reinterpret_cast<DeferList *>(smem_raw + sizeof(WSmem) + (kTen ? ten_bytes(a.H) : 0) +
                                                    (kFit ? (size_t)kWarps * 4 * fit_entries(a.fit.n_y) * sizeof(FitAcc) : 0));
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int NE4 = kFit ? 4 * fit_entries(a.fit.n_y) : 0;
  int bad = 0;

  if (kTen)
    for (int i = tid; i < 4 * ten_plane(a.H); i += kWThreads) tt[i] = 0;
  if (kFit)
    for (int i = tid; i < kWarps * NE4; i += kWThreads) facc[i] = FitAcc{{0, 0, 0, 0}};
  if ((MODE & M_ATTR) && tid < 4) ws.fx[tid] = a.mp.fx[tid];
  if (MODE & M_ATTR) {
    init_segs<MODE>(a, ws.seg);
    if (MODE & M_FIX) {
      for (int i = tid; i < 4 * (kNK + 1); i += kWThreads) {
        const int s = i / (kNK + 1), n = i % (kNK + 1);
        i128 kf = mk128(0, 0);
        bool ovf = false;
        if (n >= 1 && n <= a.mp.nk) {
          kf = a.mp.ktab[s * (a.mp.nk + 1) + n].kf;  // fix(fl(q + a4n)), built once per model
          ovf = kf.hi == kKSlowHi;
        }
        ws.kfix[s][n] = kf;
        ws.kslow[s][n] = ovf ? 1 : 0;
      }
    }
  }
  __syncthreads();

  uint8_t *owner = ws.owner[wid];
  FitAcc *fw = facc + wid * NE4;
  DeferList *dl = dlists + wid;
  uint64_t *frec = reinterpret_cast<uint64_t *>(&ws.kfix[0][0]) + wid * kFitRecs * kFitRecWords;  // fit mode only
  int dcnt = 0;
  unsigned long long t = 0;
  if (lane == 0) t = atomicAdd(a.ctr, 1ull);
  t = __shfl_sync(kFull, t, 0);
  while (t < (unsigned long long)a.n_tiles) {
    unsigned long long tn = 0;
    if (lane == 0) tn = atomicAdd(a.ctr, 1ull);  // next tile, fetched early
    const int64_t b0 = clampi(a.part[t].b, 0, a.n_batch);
    int64_t b1 = clampi(a.part[t + 1].b, b0, a.n_batch);
    if (b1 - b0 > a.D) {
      b1 = b0 + a.D;
      bad = 1;
    }
    for (int64_t g0 = b0; g0 < b1; g0 += 32)
      process_group<MODE>(a, ws, tt, owner, dl, dcnt, fw, frec, g0, (int)(b1 - g0 < 32 ? b1 - g0 : 32), lane, &bad);
    t = __shfl_sync(kFull, tn, 0);
  }
  if (MODE & M_ATTR) {
    while (dcnt > 0) dcnt = defer_flush<MODE>(a, tt, ws, *dl, dcnt, lane);
  }

  if (bad) flag(a.status, kStatusData);
  if (kTen || kFit) __syncthreads();
  if (kTen) {
    for (int u = tid; u < a.H; u += kWThreads) {
      const i128 v = hot_value(tt, a.H, u);
      if (v.lo | v.hi) pend_add(a.ten_pend, u, v);
    }
  }
  if (kFit) {
    // this CTA's partial: exact sum over its warps (flag entries ORed)
    const int NE = fit_entries(a.fit.n_y);
    for (int e = tid; e < NE4; e += kWThreads) {
      FitAcc s{{0, 0, 0, 0}};
      for (int w = 0; w < kWarps; ++w) {
        const FitAcc &v = facc[w * NE4 + e];
        if (e % NE == NE - 1)
          s.w[0] |= v.w[0];
        else
          acc_add256(s.w, v.w[0], v.w[1], v.w[2], v.w[3]);
      }
      a.fit.partial[(int64_t)blockIdx.x * NE4 + e] = s;
    }
  }
}

// Batches of more than kJumbo requests, one CTA per batch (grid-stride over
// the queue that k_warps filled).  Fit partials go to row fit_base + CTA.
template <int MODE>
__global__ void __launch_bounds__(kJBlock) k_jumbo(const TileArgs a, int fit_base) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  JSmem &js = *reinterpret_cast<JSmem *>(smem_raw);
  uint32_t *tt = reinterpret_cast<uint32_t *>(smem_raw + sizeof(JSmem));
  constexpr bool kTen = (MODE & M_TEN) != 0;
  constexpr bool kFit = (MODE & M_FIT) != 0;
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  int bad = 0;
  FitAcc facc{{0, 0, 0, 0}};
  if (kTen)
    for (int i = tid; i < 4 * ten_plane(a.H); i += kJBlock) tt[i] = 0;
  if (MODE & M_ATTR) init_segs<MODE>(a, js.seg);
  __syncthreads();

  const unsigned long long q = *a.jumbo_n;
  const int64_t nj = q < (unsigned long long)a.jumbo_cap ? (int64_t)q : a.jumbo_cap;
  for (int64_t k = blockIdx.x; k < nj; k += gridDim.x) {
    const int64_t b = clampi(a.jumbo[k], 0, a.n_batch - 1);
    const int64_t r0 = clampi(a.off[b], 0, a.n_req), r1 = clampi(a.off[b + 1], r0, a.n_req);
    Sums acc{0, 0, 0, 0};
    for (int64_t i = r0 + tid; i < r1; i += kJBlock) {
      int32_t p = a.p[i], c = a.c[i], ph = a.ph[i];
      check_req(p, c, ph, &bad);
      acc.s1 += p;
      acc.s2 += c;
      acc.s3 += (int64_t)p * p;
      acc.ph += ph;
    }
    acc = warp_sum(acc);
    if (lane == 0) js.red[wid] = acc;
    __syncthreads();
    if (tid == 0) {
      Sums t{0, 0, 0, 0};
      for (int w = 0; w < kJWarps; ++w) t = add_sums(t, js.red[w]);
      js.tot = t;
    }
    __syncthreads();
    const Sums tot = js.tot;
    const BatchAgg g{tot.s1, tot.s2, tot.s3, r1 - r0, tot.ph > 0};
    const int s = segment_of(a.mp, g);
    if (tid == 0) emit_batch<MODE>(a, b, g, s, a.mp.fx);
    if (kFit) {
      const int NE = fit_entries(a.fit.n_y);
      const int64_t x[5] = {1, g.s1, g.s2, g.s3, g.n * g.n};
      const bool in_range = g.s1 < kFitFeatMax && g.s2 < kFitFeatMax && g.s3 < kFitFeatMax && x[4] < kFitFeatMax;
      if (!in_range && tid == 0) flag(a.status, kStatusOverflow);
      if (tid < 4 * NE && tid / NE == s && in_range)
        fit_owner_add(facc, tid % NE, a.fit.n_y, x, a.fit.y, a.n_batch, b, g.s1 != g.s3, &bad);
    }
    if ((MODE & M_ATTR) && (MODE & M_F32)) {
      const Share32 q = share32_const(a.mp.coef[s], g.n);
      for (int64_t i = r0 + tid; i < r1; i += kJBlock) {
        int32_t p = a.p[i], c = a.c[i];
        p = p < 0 ? 0 : p;
        c = c < 0 ? 0 : c;
        const float sh = share_f32(q, p, c);
        if (a.share32) __stcs(a.share32 + i, sh);
        if (kTen) tenant_f32(a, tt, a.ten[i], sh, &bad);
      }
    } else if (MODE & M_ATTR) {
      bool slow = false;
      const i128 kf = batch_const_w<MODE>(a, nullptr, s, g.n, &slow);
      const SegS sg = js.seg[s];
      // decode requests through the same fast path as k_warps; the rest general
      const bool fast = (MODE & M_FIX) && !slow && sg.a2_narrow;
      const i128 K13 = add128(kf, sg.A13);
      for (int64_t i = r0 + tid; i < r1; i += kJBlock) {
        int32_t p = a.p[i], c = a.c[i];
        const int32_t u = kTen ? a.ten[i] : 0;
        p = p < 0 ? 0 : p;
        c = c < 0 ? 0 : c;
        bool done = false;
        if (fast && p == 1) {
          uint32_t v0, v1, v2, v3;
          mad_k13((uint32_t)K13.lo, (uint32_t)(K13.lo >> 32), (uint32_t)K13.hi, (uint32_t)(K13.hi >> 32),
                  (uint32_t)sg.A2.lo, (uint32_t)(sg.A2.lo >> 32), (uint32_t)c, v0, v1, v2, v3);
          if (v3 == 0u && v2 != 0u) {
            uint64_t m;
            int ex2;
            const double d = round96(v0, v1, v2, sg.E, m, ex2);
            if (!kTen || tenant_fast(a, tt, u, m, ex2)) {
              if (a.share) __stcs(a.share + i, d);
              done = true;
            }
          }
        }
        if (!done) attribute_one<MODE>(a, tt, sg, s, slow, kf, g.n, i, p, c, u, &bad);
      }
    }
    __syncthreads();  // js.red / js.tot are rewritten for the next batch
  }
  if (bad) flag(a.status, kStatusData);
  if (kFit) {
    const int NE4 = 4 * fit_entries(a.fit.n_y);
    if (tid < NE4) a.fit.partial[((int64_t)fit_base + blockIdx.x) * NE4 + tid] = facc;
  }
  if (kTen) {
    __syncthreads();
    for (int u = tid; u < a.H; u += kJBlock) {
      const i128 v = hot_value(tt, a.H, u);
      if (v.lo | v.hi) pend_add(a.ten_pend, u, v);
    }
  }
}

// ---------------------------------------------------------------- small inputs

// A serving scheduler attributes one step's batches (a few thousand requests)
// at a time, where launch latency, not bandwidth, bounds the call.  For such
// inputs lv_attribute and lv_attribute_step run this kernel instead of the
// partition, tile, jumbo, fold and totals kernels: one cluster of kStepCtas
// CTAs with one request per thread (CTA r takes the r-th contiguous share of
// the requests) and one more warp per CTA for the batch constant.  The CTAs
// exchange partial results by asynchronous stores into one another's shared
// memory, each completing bytes on the receiver's transaction barrier, so no
// step waits at a cluster-wide barrier.
//   1. Thread 0 sets up the two receive barriers (the batch sums, the tenant
//      slice), and the cluster's threads arrive once on the cluster barrier,
//      which they wait for only before their first remote store.  Every global
//      read is issued at once: the thread's request, the offsets (warp 0
//      clamps them into non-decreasing batch bounds with a max-scan), and the
//      state of the tenants this CTA folds; each CTA zeroes its tenant table.
//      The constant warp meanwhile forms the per-request constant of a batch
//      of n_req requests for all four segments (the single-batch step's).
//   2. Per-batch sums of the CTA's requests: a warp whose requests share one
//      batch (the common case) keeps its warp sums (hardware reductions when
//      they fit 31 bits), a warp that spans a batch bound adds lane by lane
//      with shared atomics.  The CTA's sums go to every CTA of the cluster.
//   3. One thread per batch adds the CTAs' partial sums as they arrive and
//      picks the segment and the constant.
//   4. Every thread attributes its request and adds its share into the CTA's
//      exact tenant table; the constant warp of CTA 0 writes T.
//   5. Tenant u's table entry goes to the CTA that owns u's slice; there one
//      thread per tenant adds the cluster's entries exactly, and the tenant's
//      state (zero on a reset) is added, stored and, when asked, converted to
//      the correctly rounded total.
// A CTA leaves only after every byte addressed to it has arrived.  Each wait
// on a receive barrier is bounded (a few seconds); one that runs out records
// a timeout in the status word.  Tenant ids from H up still go to the pending
// limbs, which the caller folds.
constexpr int kStepCtas = 8;
constexpr int kStepThreads = 512;                 // request threads
constexpr int kStepBlock = kStepThreads + 32;     // and the constant warp
constexpr int64_t kSmallMaxReq = (int64_t)kStepCtas * kStepThreads;
constexpr int64_t kSmallMaxBatch = 16;
constexpr int kStepSlice = (kHotMax + kStepCtas - 1) / kStepCtas;  // tenants a CTA folds, at most
static_assert(kSmallMaxBatch < 32, "warp 0 scans the offsets");
static_assert(kStepThreads >= kStepSlice, "one thread per tenant of a slice");
static_assert(kStepThreads >= kStepCtas * kSmallMaxBatch * 4, "one remote store per thread sends the sums");
static_assert(kStepThreads >= kHotMax, "one thread per tenant sends the table");

struct StepSmem {
  alignas(16) SegS seg[4];
  alignas(16) i128 kspec[4];                                // constant of a batch of n_req requests, per segment
  alignas(16) i128 bk[kSmallMaxBatch];                      // each batch's constant
  alignas(16) unsigned long long sum[kSmallMaxBatch][4];     // requests of warps that span a batch bound
  alignas(16) unsigned long long wsum[kStepThreads / 32][4];  // each warp's sums (warps within one batch)
  alignas(16) unsigned long long rsum[kStepCtas][kSmallMaxBatch][4];  // every CTA's, as received
  alignas(16) int64_t cb[kSmallMaxBatch + 1];               // clamped batch bounds
  alignas(8) unsigned long long mbar[2];                    // receive barriers: sums, tenant slice
  alignas(16) BatchAgg agg[kSmallMaxBatch];                 // each batch's totals
  int kspec_slow[4];
  int bs[kSmallMaxBatch], bslow[kSmallMaxBatch];
  int wb[kStepThreads / 32];                                // batch of warp wsum[w], or -1
  int pad[3];
};
static_assert(sizeof(StepSmem) % 16 == 0, "the tenant table follows StepSmem");

__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

// The address of shared-memory address `a` in the CTA of cluster rank `rank`.
__device__ __forceinline__ uint32_t peer_addr(uint32_t a, int rank) {
  uint32_t d;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(rank));
  return d;
}

// A receive barrier of one phase: one arrival (here) and `bytes` to come.
__device__ __forceinline__ void rx_init(uint32_t mb, uint32_t bytes) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mb) : "memory");
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(mb), "r"(bytes) : "memory");
}

// 8 or 16 bytes into a peer's shared memory, completing as many bytes on the
// peer's barrier `rmb`.
__device__ __forceinline__ void rx_put64(uint32_t raddr, uint64_t v, uint32_t rmb) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b64 [%0], %1, [%2];" ::"r"(raddr), "l"(v),
               "r"(rmb)
               : "memory");
}
__device__ __forceinline__ void rx_put128(uint32_t raddr, i128 v, uint32_t rmb) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];" ::"r"(
                   raddr),
               "r"((uint32_t)v.lo), "r"((uint32_t)(v.lo >> 32)), "r"((uint32_t)v.hi), "r"((uint32_t)(v.hi >> 32)),
               "r"(rmb)
               : "memory");
}

// Waits for the receive barrier's first phase (bounded: false when it ran
// out, after a few seconds); what arrived is then visible to this thread.
// Each try suspends the thread until the phase completes or about a
// microsecond has passed.
__device__ __forceinline__ bool rx_wait(uint32_t mb) {
  for (int k = 0; k < (1 << 22); ++k) {
    uint32_t done;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], 0, %2;\n"
        " selp.u32 %0, 1, 0, p;\n}"
        : "=r"(done)
        : "r"(mb), "n"(1000)
        : "memory");
    if (done) return true;
  }
  return false;
}

// This warp's contribution to the per-batch sums: when every active lane is
// in one batch (the common case), the warp's sums go to wsum[warp] (four
// hardware reductions when every sum fits 31 bits); otherwise each lane adds
// its fields to sum[its batch] with shared atomics.
__device__ __forceinline__ void step_sums(StepSmem &ss, bool at, int b, int32_t p, int32_t c, int32_t ph, int lane,
                                          int wid) {
  const unsigned am = __ballot_sync(kFull, at);
  const int b0 = am ? __shfl_sync(kFull, b, __ffs(am) - 1) : -1;
  if (__all_sync(kFull, !at || b == b0)) {
    unsigned long long w[4];
    if (__all_sync(kFull, (uint32_t)p < (1u << 13) && (uint32_t)c < (1u << 26))) {
      w[0] = __reduce_add_sync(kFull, at ? (uint32_t)p : 0u);
      w[1] = __reduce_add_sync(kFull, at ? (uint32_t)c : 0u);
      w[2] = __reduce_add_sync(kFull, at ? (uint32_t)(p * p) : 0u);
      w[3] = __reduce_add_sync(kFull, at ? (uint32_t)ph : 0u);
    } else {
      Sums v{at ? p : 0, at ? c : 0, at ? (int64_t)p * p : 0, at ? ph : 0};
      v = warp_sum(v);
      w[0] = (unsigned long long)v.s1;
      w[1] = (unsigned long long)v.s2;
      w[2] = (unsigned long long)v.s3;
      w[3] = (unsigned long long)v.ph;
    }
    if (lane == 0) {
      ss.wb[wid] = b0;
#pragma unroll
      for (int k = 0; k < 4; ++k) ss.wsum[wid][k] = w[k];
    }
  } else {
    if (lane == 0) ss.wb[wid] = -1;
    if (at) {
      atomicAdd(&ss.sum[b][0], (unsigned long long)p);
      atomicAdd(&ss.sum[b][1], (unsigned long long)c);
      atomicAdd(&ss.sum[b][2], (unsigned long long)((int64_t)p * p));
      atomicAdd(&ss.sum[b][3], (unsigned long long)ph);
    }
  }
}

// Barrier of the request threads alone (the constant warp does not wait).
__device__ __forceinline__ void sync_requests() { asm volatile("bar.sync 1, %0;" ::"n"(kStepThreads) : "memory"); }

// state: the tenant accumulator's exact state (with M_TEN); L: the tenants'
// totals after this step, or null (then tenant ids may exceed H); reset: the
// state is taken as zero.
template <int MODE>
__global__ void __cluster_dims__(kStepCtas, 1, 1) __launch_bounds__(kStepBlock)
    k_step(const TileArgs a, i128 *state, double *L, int reset) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  StepSmem &ss = *reinterpret_cast<StepSmem *>(smem_raw);
  uint32_t *tt = reinterpret_cast<uint32_t *>(smem_raw + sizeof(StepSmem));
  constexpr bool kTen = (MODE & M_TEN) != 0;
  const int TS = kTen ? (a.H + kStepCtas - 1) / kStepCtas : 0;  // tenants per slice
  i128 *rt = reinterpret_cast<i128 *>(smem_raw + sizeof(StepSmem) + (kTen ? ten_bytes(a.H) : 0));  // [src][TS]
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const int r = (int)cooperative_groups::this_cluster().block_rank();
  const int64_t nr = a.n_req, nb = a.n_batch;
  const bool req = tid < kStepThreads;
  const uint32_t mb0 = smem_u32(&ss.mbar[0]), mb1 = smem_u32(&ss.mbar[1]);
  int bad = 0;

  // 1. receive barriers, reads, the single-batch constant
  const int own = kTen ? max(0, min(TS, a.H - r * TS)) : 0;  // tenants of this CTA's slice
  if (tid == 0) {
    rx_init(mb0, (uint32_t)(kStepCtas * 32 * nb));
    rx_init(mb1, (uint32_t)(kStepCtas * 16 * own));
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory");
  const int64_t chunk = (nr + kStepCtas - 1) / kStepCtas;
  const int64_t i = r * chunk + tid;
  const bool in = req && tid < chunk && i < nr;
  int32_t p = 0, c = 0, ph = 0, u = 0;
  if (in) {
    p = a.p[i];
    c = a.c[i];
    ph = a.ph[i];
    if (kTen) u = a.ten[i];
  }
  int64_t ob = 0;
  if (wid == 0 && lane <= nb) ob = a.off[lane];
  // the fold: thread j takes tenant r * TS + j of this CTA's slice
  const int v = r * TS + tid;
  const bool fv = tid < own;
  i128 st0 = mk128(0, 0);
  if (fv && !reset) st0 = state[v];
  if (!req) {
    if (lane < 4) {
      bool slow = false;
      ss.kspec[lane] = nr > 0 ? batch_const_w<MODE>(a, nullptr, lane, nr, &slow) : mk128(0, 0);
      ss.kspec_slow[lane] = slow ? 1 : 0;
    }
  } else {
    if (kTen)
      for (int k = tid; k < 4 * ten_plane(a.H); k += kStepThreads) tt[k] = 0;
    if (tid < 4 * kSmallMaxBatch) (&ss.sum[0][0])[tid] = 0ull;
    init_segs<MODE>(a, ss.seg);
    if (in) check_req(p, c, ph, &bad);
    if (wid == 0) {
      // bound k = min(n_req, max(0, off[0..k])): batch b takes requests
      // [cb[b], cb[b + 1]); valid offsets are their own bounds
      int64_t m = lane <= nb ? max(ob, (int64_t)0) : 0;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int64_t o = __shfl_up_sync(kFull, m, d);
        if (lane >= d) m = max(m, o);
      }
      m = min(m, nr);
      if (lane <= nb) {
        ss.cb[lane] = m;
        if (r == 0 && (m != ob || (lane == 0 && ob != 0) || (lane == nb && ob != nr))) bad = 1;
      }
    }
    sync_requests();

    // 2. per-batch sums, sent to every CTA of the cluster
    int b = 0;
    for (int k = 1; k < nb; ++k) b += ss.cb[k] <= i ? 1 : 0;
    const bool at = in && i >= ss.cb[0] && i < ss.cb[nb];
    step_sums(ss, at, b, p, c, ph, lane, wid);
    sync_requests();
    asm volatile("barrier.cluster.wait;" ::: "memory");  // the peers' receive barriers are set up
    if (tid < kStepCtas * 4 * nb) {
      // word k of the CTA's batch sums (batch k / 4), to CTA dst
      const int dst = tid / (4 * (int)nb), k = tid % (4 * (int)nb), kb = k >> 2, kw = k & 3;
      unsigned long long x = ss.sum[kb][kw];
#pragma unroll
      for (int j = 0; j < kStepThreads / 32; ++j) x += ss.wb[j] == kb ? ss.wsum[j][kw] : 0ull;
      rx_put64(peer_addr(smem_u32(&ss.rsum[r][kb][kw]), dst), x, peer_addr(mb0, dst));
    }
    // each request thread keeps its batch index in p's place until step 4
    ph = at ? b : -1;
  }
  __syncthreads();

  // 3. the batches' totals, segment, T and constant
  if (tid < nb) {
    if (!rx_wait(mb0)) flag(a.status, kStatusTimeout);
    unsigned long long t[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
    for (int src = 0; src < kStepCtas; ++src)
#pragma unroll
      for (int w = 0; w < 4; ++w) t[w] += ss.rsum[src][tid][w];
    const int64_t n = ss.cb[tid + 1] - ss.cb[tid];
    const BatchAgg g{(int64_t)t[0], (int64_t)t[1], (int64_t)t[2], n, t[3] > 0};
    const int s = segment_of(a.mp, g);
    ss.agg[tid] = g;
    bool slow = false;
    i128 kf = mk128(0, 0);
    if (n == nr) {
      kf = ss.kspec[s];
      slow = ss.kspec_slow[s] != 0;
    } else if (n > 0) {
      kf = batch_const_w<MODE>(a, nullptr, s, n, &slow);
    }
    ss.bs[tid] = s;
    ss.bk[tid] = kf;
    ss.bslow[tid] = slow ? 1 : 0;
  }
  __syncthreads();

  // 4. this thread's request; T from the constant warp of CTA 0
  if (!req) {
    if (r == 0 && lane < nb) emit_batch<MODE>(a, lane, ss.agg[lane], ss.bs[lane], a.mp.fx);
  } else if (ph >= 0) {
    const int b = ph;
    const int s = ss.bs[b];
    const bool slow = ss.bslow[b] != 0;
    const i128 kf = ss.bk[b];
    const SegS sg = ss.seg[s];
    bool done = false;
    if ((MODE & M_FIX) && !slow && sg.a2_narrow && (p == 1 || (sg.p_narrow && p <= kPMaxFix))) {
      // the exact steps of the warp-tile fast path, with K + A1 + A3 for a
      // decode request and K + p (A1 + A3 p) for a prefill (one instruction
      // stream for both: a branch to rarely run code fetches it cold)
      const i128 K13 = add128(kf, sg.A13);
      uint32_t b0, b1, b2, b3, v0, v1, v2, v3;
      prefill_const(sg, kf, sg.p_narrow ? (uint32_t)p : 1u, b0, b1, b2, b3);
      if (p == 1) {
        b0 = (uint32_t)K13.lo;
        b1 = (uint32_t)(K13.lo >> 32);
        b2 = (uint32_t)K13.hi;
        b3 = (uint32_t)(K13.hi >> 32);
      }
      mad_k13(b0, b1, b2, b3, (uint32_t)sg.A2.lo, (uint32_t)(sg.A2.lo >> 32), (uint32_t)c, v0, v1, v2, v3);
      if (v3 == 0u && v2 != 0u) {
        uint64_t m;
        int ex2;
        const double d = round96(v0, v1, v2, sg.E, m, ex2);
        if (!kTen || tenant_fast(a, tt, u, m, ex2)) {
          if (a.share) __stcs(a.share + i, d);
          done = true;
        }
      }
    }
    if (!done) attribute_one<MODE>(a, tt, sg, s, slow, kf, ss.cb[b + 1] - ss.cb[b], i, p, c, u, &bad);
  }
  if (bad) flag(a.status, kStatusData);

  // 5. each tenant's table entry to the CTA of its slice, then the fold there
  if constexpr (kTen) {
    __syncthreads();
    if (tid < a.H) {
      const int dst = tid / TS;
      rx_put128(peer_addr(smem_u32(&rt[r * TS + (tid - dst * TS)]), dst), hot_value(tt, a.H, tid),
                peer_addr(mb1, dst));
    }
    if (fv) {
      if (!rx_wait(mb1)) flag(a.status, kStatusTimeout);
      i128 tv = rt[tid];
#pragma unroll
      for (int src = 1; src < kStepCtas; ++src) tv = add128(tv, rt[src * TS + tid]);
      const i128 nw = add128(st0, tv);
      // overflow of the signed 128-bit total (|total| >= 2^127 * 2^-72 s)
      if (is_neg128(st0) == is_neg128(tv) && is_neg128(nw) != is_neg128(st0)) flag(a.status, kStatusData);
      if (reset || (tv.lo | tv.hi)) state[v] = nw;
      if (L) L[v] = fix_to_double(nw, kTenLsb).d;
    }
  }
}

}  // namespace lv
