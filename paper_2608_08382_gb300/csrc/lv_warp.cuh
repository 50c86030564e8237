// Warp-level building blocks shared by the request-stream kernel
// (lv_stream.cuh) and the block-per-batch kernel k_jumbo for batches too large
// for the stream: the decode fast path of the fixed-point share, the tenant
// adds, the general path for the requests the fast path leaves, the fit
// statistics of a group of batches, and k_jumbo itself.
#pragma once

#include "lv_kernels.cuh"

namespace lv {

constexpr int kDW = 1024;                  // merge positions per warp tile (large inputs: 2 kDW)
constexpr int kJBlock = 512;               // threads per CTA of k_jumbo
constexpr int kJWarps = kJBlock / 32;
constexpr unsigned kFull = 0xffffffffu;

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

// v = k + (a1:a0) * c, four 32-bit words, exact (the sum stays below 2^128).
__device__ __forceinline__ void mad_k13(uint32_t k0, uint32_t k1, uint32_t k2, uint32_t k3, uint32_t a0, uint32_t a1,
                                        uint32_t c, uint32_t &v0, uint32_t &v1, uint32_t &v2, uint32_t &v3) {
  asm("{\n\t"
      ".reg .u32 l0, h0, l1, h1;\n\t"
      "mul.lo.u32 l0, %4, %6;\n\t"
      "mul.hi.u32 h0, %4, %6;\n\t"
      "mul.lo.u32 l1, %5, %6;\n\t"
      "mul.hi.u32 h1, %5, %6;\n\t"
      "add.cc.u32 %0, %7, l0;\n\t"
      "addc.cc.u32 %1, %8, h0;\n\t"
      "addc.cc.u32 %2, %9, 0;\n\t"
      "addc.u32 %3, %10, 0;\n\t"
      "add.cc.u32 %1, %1, l1;\n\t"
      "addc.cc.u32 %2, %2, h1;\n\t"
      "addc.u32 %3, %3, 0;\n\t"
      "}"
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

// Per-request constant of a batch from the model's K table: fixed-point K,
// or {fl(beta/n), fl(a4 n)} in fp64 mode.
template <int MODE>
__device__ __forceinline__ i128 batch_const_w(const TileArgs &a, int s, int64_t n, bool *slow) {
  if (MODE & M_FIX) return batch_k(a.mp, s, n, slow).kf;
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

// Batches too large for the request stream, one CTA per batch (grid-stride
// over the queue that k_stream filled).  Fit partials go to row fit_base + CTA.
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
      const i128 kf = batch_const_w<MODE>(a, s, g.n, &slow);
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

}  // namespace lv
