// Request-stream kernel for attribution, features and the fit (sm_103a).
//
// Every step of the path is a pass over request arrays, so the kernel is laid
// out around the request stream rather than around batches.  A warp walks a
// tile of whole batches (merge-path cut of batches + requests, k_partition)
// as a sequence of 128-request chunks: lane l holds requests 4l .. 4l+3 of the
// chunk, read with 128-bit loads, and the next chunk's loads are in flight
// while the current one is processed.  Per chunk:
//   - heads: the batch starts that fall in the chunk, from a window of 32
//     offsets (one per lane), as a 128-bit mask;
//   - sums: an in-lane then cross-lane segmented scan of (p, c, p^2, phase)
//     gives, at the last request of every batch that ends in the chunk, that
//     batch's S1, S2, S3 and prefill count (a batch that started in an
//     earlier chunk carries its running sums in);
//   - delivery: the sums go to a second window of 32 batches (one per lane),
//     where each batch's segment and per-request constant code are fixed as
//     soon as it is complete; a window whose 32 batches are all complete forms
//     T, the features or the fit statistics one batch per lane;
//   - shares: p, c and tenant of the chunk wait in a 3-chunk shared-memory
//     ring until every batch touching the chunk is complete, then each lane
//     attributes its 4 requests (one exact fixed-point share each, rounded
//     once) and writes them with two 16-byte stores.
// Batches larger than kSJ requests (k_jumbo's) are skipped by the stream.
// All sums are exact integers, so no result depends on this schedule.
#pragma once

#include <type_traits>

#include "lv_warp.cuh"

namespace lv {

constexpr int kChunk = 128;                 // requests per chunk: 32 lanes x 4 consecutive
constexpr int kRing = 3;                    // chunks held between the sums and the shares
constexpr int kSJ = 256;                    // batches of more than kSJ requests go to k_jumbo
constexpr int kCodes = 512;                 // batch codes in flight (ordinals of < 3 chunks + 1)
static_assert(kSJ <= kChunk * (kRing - 1), "an open batch never spans more chunks than the ring holds");
static_assert(kSJ <= kNK, "the per-request constant of every streamed batch is in the shared table");
static_assert(kRing * kChunk + 1 < kCodes, "codes of every chunk in the ring stay distinct");

// Per-segment values of the decode share loop: the words of A2, the scale,
// and whether A2 < 2^64 (the loop's 64 x 32-bit product).
struct SegB {
  uint32_t a0, a1;
  int E;
  int narrow;
};

// Shared memory of a k_stream CTA.
struct StreamCta {
  union {
    i128 k13[4][kNK + 1];  // fixed point: K + A13 at 2^E (the constant of a decode request's share)
    float k32[4][kNK + 1];  // fp32 variant: fl(beta/n) + fl(a4 n)
  };
  SegS seg[4];
  SegB segb[4];
  SegFix fx[4];
  float f32c[4][4];          // fp32 variant: a1, a2, a3
  uint8_t kslow[4][kNK + 4];  // 1: K outside the fixed-point range (general path)
};
static_assert(sizeof(StreamCta) % 16 == 0, "per-warp areas follow");

// One chunk in the ring: position of its first request (a multiple of 4),
// the valid range [lo, hi) within it, the head mask, and ordA, the ordinal
// such that request base + x belongs to batch ordinal ordA + (heads at <= x).
struct StreamMeta {
  int64_t base;
  int32_t lo, hi;
  uint32_t H[4];
  int32_t ordA;
  int32_t pad[3];
};

// Sums of one batch handed from the lanes holding its last request to the
// lane holding the batch.
struct Slot {
  uint64_t s1, s2, s3;
  uint32_t ph, pad;
};

// Per-warp shared memory, attribution modes.
struct WarpA {
  int4 rp[kRing][32], rc[kRing][32], ru[kRing][32];
  StreamMeta meta[kRing];
  uint16_t codes[kCodes];  // by ordinal: n << 3 | fast << 2 | segment
  Slot slot[32];
  DeferList dl;
};

// Per-warp shared memory, features and fit.
struct WarpF {
  Slot slot[32];
  uint64_t frec[kFitRecs * kFitRecWords];
};

template <int MODE>
using StreamWarp = typename std::conditional<(MODE & M_ATTR) != 0, WarpA, WarpF>::type;

// Dynamic shared memory of k_stream: CTA tables, tenant table, fit
// accumulators, then one area per warp.
template <int MODE>
__host__ __device__ constexpr size_t stream_ten_off() {
  return sizeof(StreamCta);
}
template <int MODE>
__host__ __device__ inline size_t stream_fit_off(int H) {
  return sizeof(StreamCta) + ((MODE & M_TEN) ? ten_bytes(H) : 0);
}
template <int MODE>
__host__ __device__ inline size_t stream_warp_off(int H, int n_y, int nw) {
  return stream_fit_off<MODE>(H) + ((MODE & M_FIT) ? (size_t)nw * 4 * fit_entries(n_y) * sizeof(FitAcc) : 0);
}
template <int MODE>
__host__ __device__ inline size_t stream_smem(int H, int n_y, int nw) {
  return stream_warp_off<MODE>(H, n_y, nw) + (size_t)nw * sizeof(StreamWarp<MODE>);
}

// ---------------------------------------------------------------- small helpers

// Elements i .. i+3 of a (i a multiple of 4, i >= 0); those at or beyond n
// read as 0.  One 16-byte streaming load when all four exist.
__device__ __forceinline__ int4 load4(const int32_t *__restrict__ a, int64_t i, int64_t n) {
  if (i + 4 <= n) return __ldcs(reinterpret_cast<const int4 *>(a + i));
  int4 v = make_int4(0, 0, 0, 0);
  if (i < n) v.x = a[i];
  if (i + 1 < n) v.y = a[i + 1];
  if (i + 2 < n) v.z = a[i + 2];
  return v;
}

__device__ __forceinline__ int32_t geti(const int4 &v, int t) {
  return t == 0 ? v.x : t == 1 ? v.y : t == 2 ? v.z : v.w;
}

// Bits [lo - 4 lane, hi - 4 lane) of a lane's four positions.
__device__ __forceinline__ uint32_t lane_range(int lo, int hi, int lane) {
  const int q = 4 * lane;
  const int a = min(max(lo - q, 0), 4), b = min(max(hi - q, 0), 4);
  return b > a ? (((1u << b) - 1u) & ~((1u << a) - 1u)) : 0u;
}

// This lane's four bits of a 128-bit mask held as four uniform words.
__device__ __forceinline__ uint32_t lane_nibble(const uint32_t H[4], int lane) {
  const int w = lane >> 3;
  const uint32_t x = w == 0 ? H[0] : w == 1 ? H[1] : w == 2 ? H[2] : H[3];
  return (x >> ((lane & 7) * 4)) & 0xFu;
}

// Sum over lower lanes of a per-lane count in 0..4.
__device__ __forceinline__ int excl_count4(uint32_t cnt, int lane) {
  const uint32_t lt = (1u << lane) - 1u;
  const uint32_t b0 = __ballot_sync(kFull, cnt & 1u), b1 = __ballot_sync(kFull, cnt & 2u),
                 b2 = __ballot_sync(kFull, cnt & 4u);
  return __popc(b0 & lt) + 2 * __popc(b1 & lt) + 4 * __popc(b2 & lt);
}

// ---------------------------------------------------------------- segmented sums

// Narrow quantities (every p < 2^12 and c < 2^24 in the chunk): 32-bit sums of
// at most 128 requests cannot wrap.
struct QN {
  uint32_t s1, s2, s3, ph;
};
// General quantities: 64-bit sums (S3 modulo 2^64, as the batch sums take it).
struct QW {
  uint64_t s1, s2, s3;
  uint32_t ph;
};

__device__ __forceinline__ QN qadd(const QN &a, const QN &b) { return QN{a.s1 + b.s1, a.s2 + b.s2, a.s3 + b.s3, a.ph + b.ph}; }
__device__ __forceinline__ QW qadd(const QW &a, const QW &b) { return QW{a.s1 + b.s1, a.s2 + b.s2, a.s3 + b.s3, a.ph + b.ph}; }
__device__ __forceinline__ QN qup(const QN &a, int d) {
  return QN{__shfl_up_sync(kFull, a.s1, d), __shfl_up_sync(kFull, a.s2, d), __shfl_up_sync(kFull, a.s3, d),
            __shfl_up_sync(kFull, a.ph, d)};
}
__device__ __forceinline__ QW qup(const QW &a, int d) {
  return QW{__shfl_up_sync(kFull, a.s1, d), __shfl_up_sync(kFull, a.s2, d), __shfl_up_sync(kFull, a.s3, d),
            __shfl_up_sync(kFull, a.ph, d)};
}
__device__ __forceinline__ void qzero(QN &a) { a = QN{0, 0, 0, 0}; }
__device__ __forceinline__ void qzero(QW &a) { a = QW{0, 0, 0, 0}; }
__device__ __forceinline__ QN qval(QN, int32_t p, int32_t c, int32_t ph) {
  return QN{(uint32_t)p, (uint32_t)c, (uint32_t)p * (uint32_t)p, (uint32_t)ph};
}
__device__ __forceinline__ QW qval(QW, int32_t p, int32_t c, int32_t ph) {
  return QW{(uint64_t)p, (uint64_t)c, (uint64_t)p * (uint64_t)p, (uint32_t)ph};
}
__device__ __forceinline__ Slot qslot(const QN &a) { return Slot{a.s1, a.s2, a.s3, a.ph, 0}; }
__device__ __forceinline__ Slot qslot(const QW &a) { return Slot{a.s1, a.s2, a.s3, a.ph, 0}; }

// Running sums of the batch that is open at a chunk boundary.
struct Carry {
  uint64_t s1, s2, s3;
  uint32_t ph;
};

// Segmented scan of one chunk.  p, c, ph: the lane's four requests (zero where
// invalid); h: head bits, e: end bits of the lane's positions.  For every end
// position t of this lane, s[t] is the sum over its batch's requests in this
// chunk; first bit t: the batch began before the chunk (its carry is added
// when the slot is written).
template <class Q>
__device__ __forceinline__ void chunk_scan(const int4 &P, const int4 &C, const int4 &PH, uint32_t h, int lane, Q s[4],
                                           uint32_t &first) {
  Q w[4];
  w[0] = qval(Q{}, P.x, C.x, PH.x);
  const Q v1 = qval(Q{}, P.y, C.y, PH.y), v2 = qval(Q{}, P.z, C.z, PH.z), v3 = qval(Q{}, P.w, C.w, PH.w);
  w[1] = (h & 2u) ? v1 : qadd(w[0], v1);
  w[2] = (h & 4u) ? v2 : qadd(w[1], v2);
  w[3] = (h & 8u) ? v3 : qadd(w[2], v3);
  Q x = w[3];
  int g = h != 0u;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const Q y = qup(x, d);
    const int gy = __shfl_up_sync(kFull, g, d);
    if (lane >= d) {
      if (!g) x = qadd(y, x);
      g |= gy;
    }
  }
  Q prev = qup(x, 1);
  if (lane == 0) qzero(prev);
  const bool none_left = (__ballot_sync(kFull, h != 0u) & ((1u << lane) - 1u)) == 0u;
  first = 0;
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    const bool own = (h & ((2u << t) - 1u)) != 0u;  // a head of this lane at or before t
    s[t] = own ? w[t] : qadd(prev, w[t]);
    if (!own && none_left) first |= 1u << t;
  }
}

// Slot entries for the ends ranked [r0, r0 + m) of this chunk (erank: this
// lane's first end's rank).
template <class Q>
__device__ __forceinline__ void write_slots(Slot *slot, const Q s[4], uint32_t e, uint32_t first, const Carry &cr,
                                            int erank, int r0, int m) {
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    if ((e >> t) & 1u) {
      const int r = erank + __popc(e & ((1u << t) - 1u)) - r0;
      if (r >= 0 && r < m) {
        Slot v = qslot(s[t]);
        if ((first >> t) & 1u) {
          v.s1 += cr.s1;
          v.s2 += cr.s2;
          v.s3 += cr.s3;
          v.ph += cr.ph;
        }
        slot[r] = v;
      }
    }
  }
}

// The carry after this chunk: the sums of the batch still open at its end
// (position 127 valid and not an end), else zero.
template <class Q>
__device__ __forceinline__ Carry next_carry(const Q s[4], uint32_t e, uint32_t first, const Carry &cr, bool open) {
  const Slot v = qslot(s[3]);
  const bool f = (first >> 3) & 1u;
  Carry n{v.s1 + (f ? cr.s1 : 0), v.s2 + (f ? cr.s2 : 0), v.s3 + (f ? cr.s3 : 0), v.ph + (f ? cr.ph : 0)};
  n.s1 = __shfl_sync(kFull, n.s1, 31);
  n.s2 = __shfl_sync(kFull, n.s2, 31);
  n.s3 = __shfl_sync(kFull, n.s3, 31);
  n.ph = __shfl_sync(kFull, n.ph, 31);
  (void)e;
  if (!open) n = Carry{0, 0, 0, 0};
  return n;
}

// ---------------------------------------------------------------- batch windows

// A window of up to 32 consecutive batches of the tile, batch wb + lane on
// lane `lane`: its sanitised start and end.  Offsets are clamped into
// [lo_pos, q1] and made non-decreasing (a non-monotone input records
// LV_EDATA); prev: the previous window's last end (the tile's first request
// for the first window).
struct Win {
  int64_t s, e;
  int nw;
};

__device__ __forceinline__ Win load_window(const TileArgs &a, int64_t wb, int64_t b1, int64_t prev, int64_t q1,
                                           int lane, int *bad) {
  Win w;
  w.nw = (int)(b1 - wb < 32 ? b1 - wb : 32);
  const bool act = lane < w.nw;
  const bool last = wb + w.nw == b1;  // the window holds the tile's last batch
  const int64_t x0 = act ? a.off[wb + lane] : q1;
  const int64_t x1 = act ? a.off[wb + lane + 1] : q1;
  const bool ok = !act || (x0 <= x1 && x1 <= q1 && (lane > 0 || x0 == prev) &&
                           (lane != w.nw - 1 || !last || x1 == q1));
  if (__all_sync(kFull, ok)) {
    w.s = act ? x0 : q1;
    w.e = act ? x1 : q1;
    return w;
  }
  // not a valid CSR window: record it and use contiguous, non-decreasing
  // batches instead (the first starting at prev, the tile's last ending at q1)
  *bad = 1;
  int64_t m = act ? clampi(x0, prev, q1) : q1;
  if (lane == 0) m = prev;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const int64_t y = __shfl_up_sync(kFull, m, d);
    if (lane >= d && y > m) m = y;
  }
  int64_t nx = __shfl_down_sync(kFull, m, 1);
  if (lane == w.nw - 1) nx = last ? q1 : clampi(a.off[wb + w.nw], m, q1);
  w.s = act ? m : q1;
  w.e = act ? (nx > m ? nx : m) : q1;
  return w;
}

// ---------------------------------------------------------------- deferred requests

// Attribute the first min(cnt, 32) deferred requests, one per lane, through
// the general path (the batch constant from the model's K table), move the
// rest to the front and return their number.  meta: the batch code.
template <int MODE>
__device__ __noinline__ int sdefer_flush(const TileArgs &a, uint32_t *tt, const StreamCta &cs, DeferList &L, int cnt,
                                         int lane) {
  const int take = cnt < 32 ? cnt : 32;
  if (lane < take) {
    const int code = L.meta[lane];
    const int s = code & 3;
    const int64_t n = code >> 3;
    bool slow = false;
    int bad = 0;
    const i128 kf = batch_const_w<MODE>(a, s, n, &slow);
    defer_one<MODE>(a, tt, cs.seg, s, slow, kf, n, L.q[lane], L.p[lane], L.c[lane], L.u[lane], &bad);
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
__device__ __forceinline__ void sdefer_push(const TileArgs &a, uint32_t *tt, const StreamCta &cs, DeferList &L,
                                            int &cnt, bool flag, int64_t q, int meta, int32_t p, int32_t c, int32_t u,
                                            int lane) {
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
  if (cnt >= 32) cnt = sdefer_flush<MODE>(a, tt, cs, L, cnt, lane);
}

// ---------------------------------------------------------------- the kernel

template <int MODE, int NW>
__global__ void __launch_bounds__(NW * 32, 1) k_stream(const TileArgs a) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  constexpr bool kAttr = (MODE & M_ATTR) != 0;
  constexpr bool kTen = (MODE & M_TEN) != 0;
  constexpr bool kFit = (MODE & M_FIT) != 0;
  constexpr bool kF32 = (MODE & M_F32) != 0;
  constexpr bool kFix = (MODE & M_FIX) != 0;
  using Warp = StreamWarp<MODE>;
  static_assert(!(kFit && kAttr), "fit and attribution are separate launches");

  StreamCta &cs = *reinterpret_cast<StreamCta *>(smem_raw);
  uint32_t *tt = reinterpret_cast<uint32_t *>(smem_raw + stream_ten_off<MODE>());
  const int NE = kFit ? fit_entries(a.fit.n_y) : 0;
  FitAcc *facc = reinterpret_cast<FitAcc *>(smem_raw + stream_fit_off<MODE>(a.H));
  const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  Warp &W = reinterpret_cast<Warp *>(smem_raw + stream_warp_off<MODE>(a.H, a.fit.n_y, NW))[wid];
  int bad = 0;

  // ---- CTA tables
  if (kTen)
    for (int i = tid; i < 4 * ten_plane(a.H); i += NW * 32) tt[i] = 0;
  if (kFit)
    for (int i = tid; i < NW * 4 * NE; i += NW * 32) facc[i] = FitAcc{{0, 0, 0, 0}};
  if (tid < 4) {
    cs.fx[tid] = a.mp.fx[tid];
    const SegFix &f = a.mp.fx[tid];
    cs.segb[tid] = SegB{(uint32_t)f.A2.lo, (uint32_t)(f.A2.lo >> 32), f.E, f.a2_narrow};
    if (kF32) {
      const Share32 q = share32_const(a.mp.coef[tid], 1);
      cs.f32c[tid][0] = q.a1;
      cs.f32c[tid][1] = q.a2;
      cs.f32c[tid][2] = q.a3;
      cs.f32c[tid][3] = 0.0f;
    }
  }
  if (kAttr) {
    init_segs<MODE>(a, cs.seg);
    for (int i = tid; i < 4 * (kNK + 1); i += NW * 32) {
      const int s = i / (kNK + 1), n = i % (kNK + 1);
      if (kF32) {
        cs.k32[s][n] = n >= 1 ? share32_const(a.mp.coef[s], n).K : 0.0f;
        cs.kslow[s][n] = 0;
      } else {
        i128 kf = mk128(0, 0);
        bool slow = !kFix;
        if (kFix && n >= 1 && n <= a.mp.nk) {
          kf = a.mp.ktab[s * (a.mp.nk + 1) + n].kf;  // fix(fl(q + a4n)), built once per model
          slow = kf.hi == kKSlowHi;
        }
        cs.k13[s][n] = slow ? mk128(0, 0) : add128(kf, a.mp.fx[s].A13);
        cs.kslow[s][n] = slow ? 1 : 0;
      }
    }
  }
  __syncthreads();

  FitAcc *fw = kFit ? facc + wid * 4 * NE : nullptr;
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
    if (b1 > b0) {
      const int64_t q0 = clampi(a.off[b0], 0, a.n_req);
      const int64_t q1 = clampi(a.off[b1], q0, a.n_req);

      // ---- mark cursor: batch starts, for the head masks and the stream layout
      int64_t mb = b0;
      Win mw = load_window(a, mb, b1, q0, q1, lane, &bad);
      int mcons = 0;   // lanes of the mark window already placed
      int mord = 0;    // non-empty streamed batches marked so far

      // ---- delivery window: batches waiting for their sums
      int64_t db = b0;
      Win dw = load_window(a, db, b1, q0, q1, lane, &bad);
      bool ddone;
      int dord;
      int dord_next = 0;
      Sums ds{0, 0, 0, 0};
      auto open_window = [&]() {
        const int64_t n = dw.e - dw.s;
        const bool act = lane < dw.nw;
        const bool jumbo = act && n > kSJ;
        ddone = !act || n == 0 || jumbo;
        if (jumbo) {
          const unsigned long long slot = atomicAdd(a.jumbo_n, 1ull);
          if (slot < (unsigned long long)a.jumbo_cap)
            a.jumbo[slot] = db + lane;
          else
            bad = 1;
        }
        const uint32_t sm = __ballot_sync(kFull, act && n > 0 && !jumbo);
        dord = dord_next + __popc(sm & ((1u << lane) - 1u));
        dord_next += __popc(sm);
        ds = Sums{0, 0, 0, 0};
      };
      open_window();
      bool dfinished = false;

      // window epilogue: T, features, fit statistics of its batches, one per lane
      auto close_window = [&]() {
        const int64_t n = dw.e - dw.s;
        const bool act = lane < dw.nw;
        int fseg = -1;
        if (act && n <= kSJ) {
          const BatchAgg g{ds.s1, ds.s2, ds.s3, n, ds.ph > 0};
          const int s = segment_of(a.mp, g);
          emit_batch<MODE>(a, db + lane, g, s, cs.fx);
          if (kFit) {
            const bool in_range = g.s1 < kFitFeatMax && g.s2 < kFitFeatMax && g.s3 < kFitFeatMax &&
                                  n * n < kFitFeatMax;
            if (!in_range) flag(a.status, kStatusOverflow);
            if (n > 0 && in_range) fseg = s;
          }
        }
        if (kFit) {
          if constexpr (kFit) fit_group(a, fw, W.frec, db, ds, n, fseg, lane, &bad);
        }
      };

      // advance the delivery window over complete windows
      auto advance = [&]() {
        while (!dfinished && __all_sync(kFull, ddone)) {
          close_window();
          const int64_t prev = __shfl_sync(kFull, dw.e, dw.nw - 1);
          db += dw.nw;
          if (db >= b1) {
            dfinished = true;
            break;
          }
          dw = load_window(a, db, b1, prev, q1, lane, &bad);
          open_window();
        }
      };
      advance();

      // ---- the stream
      int64_t base = q0 & ~(int64_t)3;
      int lo = (int)(q0 - base);
      Carry carry{0, 0, 0, 0};
      int4 P, C, PH, U = make_int4(0, 0, 0, 0);
      P = load4(a.p, base + 4 * lane, a.n_req);
      C = load4(a.c, base + 4 * lane, a.n_req);
      PH = load4(a.ph, base + 4 * lane, a.n_req);
      if (kTen) U = load4(a.ten, base + 4 * lane, a.n_req);
      int rk = 0, rb = 0;  // ring: chunks written, chunks attributed

      // B: shares of ring chunk rb
      auto shares = [&](int r) {
        if constexpr (kAttr) {
          const int slot = r % kRing;
          const StreamMeta M = W.meta[slot];
          const int4 Pr = W.rp[slot][lane], Cr = W.rc[slot][lane];
          int4 Ur = make_int4(0, 0, 0, 0);
          if (kTen) Ur = W.ru[slot][lane];
          const uint32_t vm = lane_range(M.lo, M.hi, lane);
          const uint32_t h = lane_nibble(M.H, lane);
          const int hb = excl_count4(__popc(h), lane);
          const int64_t q = M.base + 4 * lane;
          if (kF32) {
            float res[4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const int ord = M.ordA + hb + __popc(h & ((2u << t) - 1u));
              const int code = W.codes[ord & (kCodes - 1)];
              const int s = code & 3, n = min(code >> 3, kNK);
              const Share32 sq{cs.k32[s][n], cs.f32c[s][0], cs.f32c[s][1], cs.f32c[s][2]};
              res[t] = share_f32(sq, geti(Pr, t), geti(Cr, t));
              if (kTen && ((vm >> t) & 1u)) tenant_f32(a, tt, geti(Ur, t), res[t], &bad);
            }
            if (a.share32) {
              if (vm == 0xFu && (reinterpret_cast<uintptr_t>(a.share32) & 15u) == 0) {
                __stcs(reinterpret_cast<float4 *>(a.share32 + q), make_float4(res[0], res[1], res[2], res[3]));
              } else {
#pragma unroll
                for (int t = 0; t < 4; ++t)
                  if ((vm >> t) & 1u) __stcs(a.share32 + q + t, res[t]);
              }
            }
          } else {
            double res[4];
            uint32_t okm = 0;
            int codes[4];
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const int ord = M.ordA + hb + __popc(h & ((2u << t) - 1u));
              const int code = W.codes[ord & (kCodes - 1)];
              codes[t] = code;
              res[t] = 0.0;
              if (kFix) {
                const int s = code & 3, n = min(code >> 3, kNK);
                const i128 K13 = cs.k13[s][n];
                const SegB sb = cs.segb[s];
                uint32_t v0, v1, v2, v3;
                mad_k13((uint32_t)K13.lo, (uint32_t)(K13.lo >> 32), (uint32_t)K13.hi, (uint32_t)(K13.hi >> 32), sb.a0,
                        sb.a1, (uint32_t)geti(Cr, t), v0, v1, v2, v3);
                uint64_t m;
                int ex2;
                res[t] = round96(v0, v1, v2, sb.E, m, ex2);
                bool ok = ((vm >> t) & 1u) && (code & 4) && geti(Pr, t) == 1 && v3 == 0u && v2 != 0u;
                if (kTen && ok) ok = tenant_fast(a, tt, geti(Ur, t), m, ex2);
                okm |= ok ? (1u << t) : 0u;
              }
            }
            if (a.share) {
              // 16-byte stores where the output array allows them (it need only be 8-byte aligned)
              if (okm == 0xFu && (reinterpret_cast<uintptr_t>(a.share) & 15u) == 0) {
                double2 *d = reinterpret_cast<double2 *>(a.share + q);
                __stcs(d, make_double2(res[0], res[1]));
                __stcs(d + 1, make_double2(res[2], res[3]));
              } else {
#pragma unroll
                for (int t = 0; t < 4; ++t)
                  if ((okm >> t) & 1u) __stcs(a.share + q + t, res[t]);
              }
            }
            // requests the fast loop does not cover: 32 at a time through the general path
#pragma unroll
            for (int t = 0; t < 4; ++t) {
              const bool dfl = ((vm >> t) & 1u) && !((okm >> t) & 1u);
              sdefer_push<MODE>(a, tt, cs, W.dl, dcnt, dfl, q + t, codes[t], geti(Pr, t), geti(Cr, t), geti(Ur, t),
                                lane);
            }
          }
        }
        (void)r;
      };

      while (true) {
        // ---- marking: heads of this chunk, its valid end, where the next chunk starts
        uint32_t H[4] = {0u, 0u, 0u, 0u};
        int hi = (int)min((int64_t)kChunk, q1 - base);
        if (hi < lo) hi = lo;
        const int ordA = mord - 1;
        bool jumped = false;
        int64_t nstart = base + kChunk;  // first request of the next chunk's valid range
        while (true) {
          const bool act = lane >= mcons && lane < mw.nw;
          const bool cand = act && mw.s < base + kChunk;
          const bool jmb = cand && mw.e - mw.s > kSJ;
          uint32_t cm = __ballot_sync(kFull, cand);
          const uint32_t jm = __ballot_sync(kFull, jmb);
          int jf = 32;
          if (jm) {
            jf = __ffs(jm) - 1;
            cm &= (1u << jf) - 1u;
          }
          const bool mk = ((cm >> lane) & 1u) && mw.e > mw.s;
          const int rel = (int)(mw.s - base);
#pragma unroll
          for (int w = 0; w < 4; ++w)
            H[w] |= __reduce_or_sync(kFull, (mk && (rel >> 5) == w) ? (1u << (rel & 31)) : 0u);
          mord += __popc(__ballot_sync(kFull, mk));
          if (jm) {
            const int64_t js = __shfl_sync(kFull, mw.s, jf), je = __shfl_sync(kFull, mw.e, jf);
            hi = (int)(js - base);
            if (hi < lo) hi = lo;
            nstart = je;
            jumped = true;
            mcons = jf + 1;
          } else {
            mcons += __popc(cm);
          }
          if (mcons < mw.nw) break;
          // window used up: the next one (its first batches may start in this chunk too)
          const int64_t prev = __shfl_sync(kFull, mw.e, mw.nw - 1);
          mb += mw.nw;
          if (mb >= b1) {
            mw.nw = 0;
            mcons = 0;
            break;
          }
          mw = load_window(a, mb, b1, prev, q1, lane, &bad);
          mcons = 0;
          if (jumped) break;
        }
        // position base + 128 starts a batch (or ends the tile): position 127 ends one
        bool bound128 = false;
        if (!jumped && hi == kChunk) {
          if (mcons < mw.nw)
            bound128 = __shfl_sync(kFull, mw.s, mcons) == base + kChunk;
          else
            bound128 = q1 == base + kChunk;
        }
        const bool more = nstart < q1;
        const int64_t nbase = nstart & ~(int64_t)3;

        // ---- next chunk's loads
        int4 P2 = make_int4(0, 0, 0, 0), C2 = P2, PH2 = P2, U2 = P2;
        if (more) {
          P2 = load4(a.p, nbase + 4 * lane, a.n_req);
          C2 = load4(a.c, nbase + 4 * lane, a.n_req);
          PH2 = load4(a.ph, nbase + 4 * lane, a.n_req);
          if (kTen) U2 = load4(a.ten, nbase + 4 * lane, a.n_req);
        }

        if (hi > lo) {
          // ---- validity, clamping
          const uint32_t vm = lane_range(lo, hi, lane);
          int pv[4] = {P.x, P.y, P.z, P.w}, cv[4] = {C.x, C.y, C.z, C.w}, hv[4] = {PH.x, PH.y, PH.z, PH.w};
          uint32_t por = 0, cor = 0;
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            if ((vm >> t) & 1u) {
              check_req(pv[t], cv[t], hv[t], &bad);
            } else {
              pv[t] = cv[t] = hv[t] = 0;
            }
            por |= (uint32_t)pv[t];
            cor |= (uint32_t)cv[t];
          }
          const int4 Pc = make_int4(pv[0], pv[1], pv[2], pv[3]), Cc = make_int4(cv[0], cv[1], cv[2], cv[3]),
                     Hc = make_int4(hv[0], hv[1], hv[2], hv[3]);
          if constexpr (kAttr) {
            const int slot = rk % kRing;
            W.rp[slot][lane] = Pc;
            W.rc[slot][lane] = Cc;
            if (kTen) W.ru[slot][lane] = U;
            if (lane == 0) {
              StreamMeta M;
              M.base = base;
              M.lo = lo;
              M.hi = hi;
              M.H[0] = H[0];
              M.H[1] = H[1];
              M.H[2] = H[2];
              M.H[3] = H[3];
              M.ordA = ordA;
              M.pad[0] = M.pad[1] = M.pad[2] = 0;
              W.meta[slot] = M;
            }
          }
          ++rk;
          // ---- heads and ends of this lane's positions
          const uint32_t h = lane_nibble(H, lane);
          uint32_t hn = __shfl_down_sync(kFull, h, 1);
          if (lane == 31) hn = bound128 ? 1u : 0u;
          uint32_t e = ((h >> 1) | ((hn & 1u) << 3)) & vm;
          if (hi < kChunk && ((hi - 1) >> 2) == lane) e |= 1u << ((hi - 1) & 3);
          const int erank = excl_count4(__popc(e), lane);
          // ---- sums
          const bool narrow = __all_sync(kFull, (por >> 12) == 0u && (cor >> 24) == 0u);
          uint32_t first = 0;
          QN sn[4];
          QW sw[4];
          if (narrow)
            chunk_scan<QN>(Pc, Cc, Hc, h, lane, sn, first);
          else
            chunk_scan<QW>(Pc, Cc, Hc, h, lane, sw, first);
          // ---- delivery to the windows whose batches end here
          int r0 = 0;
          while (!dfinished) {
            const bool fin = !ddone && dw.e - 1 >= base + lo && dw.e - 1 < base + hi;
            const uint32_t fm = __ballot_sync(kFull, fin);
            if (fm) {
              const int m = __popc(fm);
              __syncwarp();
              if (narrow)
                write_slots<QN>(W.slot, sn, e, first, carry, erank, r0, m);
              else
                write_slots<QW>(W.slot, sw, e, first, carry, erank, r0, m);
              __syncwarp();
              if (fin) {
                const Slot v = W.slot[__popc(fm & ((1u << lane) - 1u))];
                ds = Sums{(int64_t)v.s1, (int64_t)v.s2, (int64_t)v.s3, (int32_t)v.ph};
                ddone = true;
                if constexpr (kAttr) {
                  const int64_t n = dw.e - dw.s;
                  const BatchAgg g{ds.s1, ds.s2, ds.s3, n, ds.ph > 0};
                  const int s = segment_of(a.mp, g);
                  int fast = 0;
                  if (kFix) fast = !cs.kslow[s][n] && cs.segb[s].narrow;
                  W.codes[dord & (kCodes - 1)] = (uint16_t)((n << 3) | (fast << 2) | s);
                }
              }
              r0 += m;
            }
            if (!__all_sync(kFull, ddone)) break;
            advance();
          }
          // ---- carry into the next chunk
          const bool open = hi == kChunk && !((__shfl_sync(kFull, e, 31) >> 3) & 1u);
          if (narrow)
            carry = next_carry<QN>(sn, e, first, carry, open);
          else
            carry = next_carry<QW>(sw, e, first, carry, open);
        } else {
          carry = Carry{0, 0, 0, 0};
          advance();
        }

        // ---- shares of every ring chunk whose batches are all complete
        if constexpr (kAttr) {
          int64_t frontier = q1;
          if (!dfinished) {
            const uint32_t nd = __ballot_sync(kFull, !ddone);
            if (nd) frontier = __shfl_sync(kFull, dw.s, __ffs(nd) - 1);
          }
          while (rb < rk) {
            const StreamMeta &M = W.meta[rb % kRing];
            const bool ready = M.base + M.hi <= frontier;
            if (!ready && rk - rb < kRing) break;
            if (!ready) bad = 1;  // cannot happen for valid input: every open batch fits the ring
            shares(rb);
            ++rb;
          }
        }
        if (!more) break;
        base = nbase;
        lo = (int)(nstart - nbase);
        P = P2;
        C = C2;
        PH = PH2;
        U = U2;
      }
      // every batch of the tile is complete now
      advance();
      if (!dfinished) bad = 1;
      if constexpr (kAttr) {
        while (rb < rk) {
          shares(rb);
          ++rb;
        }
      }
    }
    t = __shfl_sync(kFull, tn, 0);
  }
  if constexpr (kAttr) {
    if (!kF32)
      while (dcnt > 0) dcnt = sdefer_flush<MODE>(a, tt, cs, W.dl, dcnt, lane);
  }

  if (bad) flag(a.status, kStatusData);
  if (kTen || kFit) __syncthreads();
  if (kTen) {
    for (int u = tid; u < a.H; u += NW * 32) {
      const i128 v = hot_value(tt, a.H, u);
      if (v.lo | v.hi) pend_add(a.ten_pend, u, v);
    }
  }
  if constexpr (kFit) {
    // this CTA's partial: exact sum over its warps (flag entries ORed)
    const int NE4 = 4 * NE;
    for (int e = tid; e < NE4; e += NW * 32) {
      FitAcc s{{0, 0, 0, 0}};
      for (int w = 0; w < NW; ++w) {
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

}  // namespace lv
