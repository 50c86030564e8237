// Host side of the C ABI declared in include/llmvisor.h: contexts, argument
// validation, fixed-point parameter derivation and kernel launch sequences.
#include <cuda_runtime.h>

#include <cmath>
#include <cstddef>
#include <mutex>
#include <cstdint>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

#include "llmvisor.h"
#include "lv_fit.cuh"
#include "lv_kernels.cuh"
#include "lv_metrics.cuh"
#include "lv_warp.cuh"
#include "lv_whatif.cuh"

using namespace lv;

struct lv_ctx {
  int device = 0;
  int sms = 0;
  int arith = LV_ARITH_AUTO;
  int *d_status = nullptr;
  TilePart *d_tiles = nullptr;
  int64_t tiles_cap = 0;
  unsigned long long *d_ctr = nullptr;  // [0] warp tiles handed out, [1] jumbo batches queued
  int64_t *d_jumbo = nullptr;
  int64_t jumbo_cap = 0;
  KEntry *d_ktab = nullptr;
  int ktab_nk = 0;
  bool ktab_valid = false;
  lv_model ktab_model{};
  int ktab_fixed = -1;
  cudaEvent_t ev_built = nullptr;
  cudaEvent_t ev_used = nullptr;
  cudaStream_t ktab_stream = nullptr;
  void *d_fit = nullptr;      // fit partials + solve output
  size_t fit_cap = 0;
  int64_t last_grid = 0;      // CTAs of the most recent tile-kernel launch
  std::vector<std::pair<uint64_t, int>> occ;  // (mode << 32 | dynamic smem) -> k_warps CTAs per SM
  void *d_wi = nullptr;       // what-if per-candidate / per-pending tables
  size_t wi_cap = 0;
  void *d_acc = nullptr;      // accuracy metrics: relative-error bits, partials, histograms
  size_t acc_cap = 0;
  int acc_occ = 0;            // CTAs per SM of the accuracy kernel (0: not yet queried)
  double *h_acc = nullptr;    // accuracy results: pinned host memory the kernel writes (mapped)
  double *hd_acc = nullptr;   // its device address
  void *d_probe = nullptr;    // barrier self-test: arrivals, generation, error word
  int timing = 0;  // LV_TIME_* mask
  std::vector<cudaEvent_t> tev;  // start/stop pairs
  size_t tev_used = 0;
};

struct lv_tenant_acc {
  lv_ctx *ctx = nullptr;
  int32_t n_tenants = 0;
  unsigned long long *d_pend = nullptr;  // [n][4]
  i128 *d_state = nullptr;               // [n]
};

namespace {

constexpr int kKTableN = 4096;

#define LV_CUDA(call)                          \
  do {                                         \
    if ((call) != cudaSuccess) return LV_ECUDA; \
  } while (0)

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

int lsb_exp(double x) {
  // x = M * 2^e with M odd; returns e.  x != 0, finite.
  int e;
  const double f = std::frexp(std::fabs(x), &e);  // x = f * 2^e, 0.5 <= f < 1
  uint64_t M = (uint64_t)std::ldexp(f, 53);
  int ex = e - 53;
  while ((M & 1ull) == 0) {
    M >>= 1;
    ++ex;
  }
  return ex;
}

int msb_exp(double x) {
  int e;
  std::frexp(std::fabs(x), &e);
  return e - 1;
}

i128 host_fix_exact(double x, int E, bool *ok) {
  bool ovf = false;
  i128 r = double_to_fix(x, E, &ovf);
  if (ovf) *ok = false;
  return r;
}

// |A| as a double (for bound checks).
double mag(i128 a) {
  if (is_neg128(a)) a = neg128(a);
  return std::ldexp((double)a.hi, 64) + (double)a.lo;
}

uint64_t limit_for(i128 A) {
  const double m = mag(A);
  if (m == 0) return (uint64_t)INT64_MAX;
  const double lim = std::floor(std::ldexp(1.0, 124) / m);
  if (lim >= 9.2e18) return (uint64_t)INT64_MAX;
  return (uint64_t)lim;
}

bool finite_model(const lv_model *m) {
  const double *c = &m->seg[0][0].beta;
  for (int i = 0; i < 20; ++i)
    if (!std::isfinite(c[i])) return false;
  return true;
}

// Derives the exact fixed-point representation of every segment.  Returns
// false when some segment's coefficients do not fit the integer path.
bool derive_fixed(const lv_model *m, int nk, ModelP *mp) {
  for (int s = 0; s < 4; ++s) {
    const lv_coef &k = m->seg[s >> 1][s & 1];
    int E = INT32_MAX;
    const double slopes[4] = {k.a1, k.a2, k.a3, k.a4};
    for (double v : slopes)
      if (v != 0) E = std::min(E, lsb_exp(v));
    if (k.beta != 0) E = std::min(E, msb_exp(k.beta) - 66);
    if (E == INT32_MAX) E = -200;  // all-zero segment: any scale works
    if (E < -1022 || E + 127 > 1023) return false;
    SegFix &f = mp->fx[s];
    std::memset(&f, 0, sizeof(f));
    f.E = E;
    bool ok = true;
    f.A1 = host_fix_exact(k.a1, E, &ok);
    f.A2 = host_fix_exact(k.a2, E, &ok);
    f.A3 = host_fix_exact(k.a3, E, &ok);
    f.B = host_fix_exact(k.beta, E, &ok);
    f.A4 = host_fix_exact(k.a4, E, &ok);
    if (!ok) return false;
    // share path: every term below 2^124 for p <= 2^24, c < 2^31
    if (mag(f.A1) >= std::ldexp(1.0, 100) || mag(f.A2) >= std::ldexp(1.0, 93) || mag(f.A3) >= std::ldexp(1.0, 76))
      return false;
    const double kmax = (std::fabs(k.beta) + std::fabs(k.a4) * nk) * 1.0000001;
    if (std::ldexp(kmax, -E) >= std::ldexp(1.0, 123) || mag(f.B) >= std::ldexp(1.0, 124)) return false;
    f.A13 = add128(f.A1, f.A3);
    f.a2_narrow = (f.A2.hi == 0) ? 1 : 0;
    f.t_narrow = (f.B.hi | f.A1.hi | f.A2.hi | f.A3.hi | f.A4.hi) < (1ull << 32) ? 1 : 0;
    f.pad = 0;
    f.lim[0] = limit_for(f.A1);
    f.lim[1] = limit_for(f.A2);
    f.lim[2] = limit_for(f.A3);
    f.lim[3] = limit_for(f.A4);
  }
  return true;
}

lv_status check_model(const lv_model *m) {
  if (!m) return LV_EINVAL;
  if (!finite_model(m)) return LV_EINVAL;
  return LV_OK;
}

lv_status check_batches(const lv_batches *b, bool need_tenant) {
  if (!b) return LV_EINVAL;
  if (b->n_req < 0 || b->n_batch < 0) return LV_EINVAL;
  if (!b->offsets || !aligned(b->offsets, 16)) return LV_EINVAL;
  if (b->n_req > 0) {
    if (!b->p || !b->c || !b->phase) return LV_EINVAL;
    if (!aligned(b->p, 16) || !aligned(b->c, 16) || !aligned(b->phase, 16)) return LV_EINVAL;
    if (need_tenant && (!b->tenant || !aligned(b->tenant, 16))) return LV_EINVAL;
  }
  if (need_tenant && b->n_tenants <= 0) return LV_EINVAL;
  if (b->n_req > (1ll << 40) || b->n_batch > (1ll << 40)) return LV_EINVAL;
  return LV_OK;
}

lv_status ensure_tiles(lv_ctx *ctx, int64_t n) {
  if (n <= ctx->tiles_cap) return LV_OK;
  LV_CUDA(cudaDeviceSynchronize());
  if (ctx->d_tiles) cudaFree(ctx->d_tiles);
  ctx->d_tiles = nullptr;
  int64_t cap = std::max<int64_t>(n, 1 << 16);
  if (cudaMalloc(&ctx->d_tiles, cap * sizeof(TilePart)) != cudaSuccess) {
    ctx->tiles_cap = 0;
    return LV_ENOMEM;
  }
  ctx->tiles_cap = cap;
  return LV_OK;
}

// Builds (or reuses) the per-model parameters and K table on `stream`.
// Event record and wait that stay valid while `stream` is being captured into a
// CUDA graph: the graph then records (waits for) the event itself at every
// replay, so a captured call still orders itself after the context's earlier
// work on other streams, and later calls after the replay.
bool capturing(cudaStream_t stream) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  return cudaStreamIsCapturing(stream, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive;
}

lv_status record_event(cudaEvent_t ev, cudaStream_t stream) {
  LV_CUDA(cudaEventRecordWithFlags(ev, stream, capturing(stream) ? cudaEventRecordExternal : cudaEventRecordDefault));
  return LV_OK;
}

lv_status wait_event(cudaStream_t stream, cudaEvent_t ev) {
  LV_CUDA(cudaStreamWaitEvent(stream, ev, capturing(stream) ? cudaEventWaitExternal : cudaEventWaitDefault));
  return LV_OK;
}

// Per-model launch parameters, formed on the host (no K table).
void model_params(const lv_ctx *ctx, const lv_model *m, ModelP *mp) {
  std::memset(mp, 0, sizeof(*mp));
  for (int s = 0; s < 4; ++s) {
    const lv_coef &k = m->seg[s >> 1][s & 1];
    mp->coef[s][0] = k.beta;
    mp->coef[s][1] = k.a1;
    mp->coef[s][2] = k.a2;
    mp->coef[s][3] = k.a3;
    mp->coef[s][4] = k.a4;
  }
  mp->split[0] = m->split[0];
  mp->split[1] = m->split[1];
  mp->nk = kKTableN;
  mp->fixed = 0;
  if (ctx->arith == LV_ARITH_AUTO) mp->fixed = derive_fixed(m, kKTableN, mp) ? 1 : 0;
}

lv_status prepare_model(lv_ctx *ctx, const lv_model *m, cudaStream_t stream, ModelP *mp) {
  model_params(ctx, m, mp);
  if (!ctx->d_ktab) {
    if (cudaMalloc(&ctx->d_ktab, sizeof(KEntry) * 4 * (kKTableN + 1)) != cudaSuccess) return LV_ENOMEM;
  }
  mp->ktab = ctx->d_ktab;
  const bool same = ctx->ktab_valid && ctx->ktab_fixed == mp->fixed &&
                    std::memcmp(&ctx->ktab_model, m, sizeof(lv_model)) == 0;
  if (!same) {
    // wait for earlier users of the table on any stream
    lv_status st = wait_event(stream, ctx->ev_used);
    if (st != LV_OK) return st;
    const int n = 4 * (kKTableN + 1);
    k_ktable<<<(n + 255) / 256, 256, 0, stream>>>(*mp, ctx->d_ktab);
    LV_CUDA(cudaGetLastError());
    st = record_event(ctx->ev_built, stream);
    if (st != LV_OK) return st;
    ctx->ktab_model = *m;
    ctx->ktab_fixed = mp->fixed;
    ctx->ktab_valid = true;
    ctx->ktab_stream = stream;
  } else if (stream != ctx->ktab_stream) {
    lv_status st = wait_event(stream, ctx->ev_built);
    if (st != LV_OK) return st;
  }
  return LV_OK;
}

// Event pair around a measured launch (when timing is on; not while the stream
// is being captured into a graph).
lv_status timing_begin(lv_ctx *ctx, int kind, cudaStream_t stream, cudaEvent_t *stop) {
  *stop = nullptr;
  if (!(ctx->timing & kind) || capturing(stream)) return LV_OK;
  if (ctx->tev_used + 2 > ctx->tev.size()) {
    for (int k = 0; k < 2; ++k) {
      cudaEvent_t e;
      LV_CUDA(cudaEventCreate(&e));
      ctx->tev.push_back(e);
    }
  }
  cudaEvent_t start = ctx->tev[ctx->tev_used];
  *stop = ctx->tev[ctx->tev_used + 1];
  ctx->tev_used += 2;
  LV_CUDA(cudaEventRecord(start, stream));
  return LV_OK;
}

lv_status timing_end(cudaEvent_t stop, cudaStream_t stream) {
  if (stop) LV_CUDA(cudaEventRecord(stop, stream));
  return LV_OK;
}

// Dynamic shared memory of k_warps for a tenant table of H entries and n_y fit vectors.
template <int MODE>
size_t warps_smem(int H, int n_y) {
  return sizeof(WSmem) + ((MODE & M_TEN) ? ten_bytes(H) : 0) +
         ((MODE & M_FIT) ? (size_t)kWarps * 4 * fit_entries(n_y) * sizeof(FitAcc) : 0) +
         ((MODE & M_ATTR) ? (size_t)kWarps * sizeof(DeferList) : 0);
}

constexpr int kJumboCtasPerSm = 2;

// Occupancy of k_warps<MODE> for launches without a context, by (mode << 32 |
// dynamic shared memory); the kernel attributes are process-wide as well.
template <int MODE>
std::vector<std::pair<uint64_t, int>> &free_occ() {
  static std::vector<std::pair<uint64_t, int>> v;
  return v;
}
template <int MODE>
std::mutex &free_occ_mu() {
  static std::mutex m;
  return m;
}

// Upper bound on the CTAs of one k_warps + k_jumbo pair (rows of fit partials).
int64_t max_tile_ctas(int sms) { return (int64_t)sms * (2048 / kWThreads + kJumboCtasPerSm); }

// k_warps then k_jumbo for the partitioned batches in `a` (a.part, a.ctr,
// a.jumbo* set, counters zeroed on `stream`).  *ctas receives the number of
// CTAs launched (fit partial rows).  ctx may be null (no timing).
template <int MODE>
lv_status launch_warps_mode(lv_ctx *ctx, int sms, TileArgs &a, cudaStream_t stream, int64_t *ctas) {
  *ctas = 0;
  const size_t smem = warps_smem<MODE>(a.H, a.fit.n_y);
  const size_t jsmem = sizeof(JSmem) + ((MODE & M_TEN) ? ten_bytes(a.H) : 0);
  const uint64_t key = ((uint64_t)MODE << 32) | smem;
  int per_sm = 0;
  if (ctx) {
    for (const auto &e : ctx->occ)
      if (e.first == key) per_sm = e.second;
  } else {
    // context-free callers (lv_attribute_noalloc): a process-wide cache per mode
    std::lock_guard<std::mutex> lock(free_occ_mu<MODE>());
    for (const auto &e : free_occ<MODE>())
      if (e.first == key) per_sm = e.second;
  }
  if (per_sm == 0) {
    // kernel attributes and occupancy: once per (context, mode, shared-memory size)
    LV_CUDA(cudaFuncSetAttribute(k_warps<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)warps_smem<MODE>(kHotMax, kFitMaxY)));
    LV_CUDA(cudaFuncSetAttribute(k_jumbo<MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(sizeof(JSmem) + ten_bytes(kHotMax))));
    LV_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_warps<MODE>, kWThreads, smem));
    if (per_sm < 1) per_sm = 1;
    if (ctx) {
      ctx->occ.emplace_back(key, per_sm);
    } else {
      std::lock_guard<std::mutex> lock(free_occ_mu<MODE>());
      free_occ<MODE>().emplace_back(key, per_sm);
    }
  }
  const int64_t grid = std::min<int64_t>(a.n_tiles, (int64_t)sms * per_sm);
  if (grid <= 0) return LV_OK;
  // k_jumbo: at most one CTA per batch that can exceed kJumbo requests (none
  // for small inputs, e.g. a single serving step of a few hundred requests)
  const int64_t jgrid = std::min<int64_t>((int64_t)sms * kJumboCtasPerSm, a.n_req / (kJumbo + 1));
  cudaEvent_t stop = nullptr;
  if (ctx) {
    lv_status st = timing_begin(ctx, LV_TIME_TILES, stream, &stop);
    if (st != LV_OK) return st;
  }
  k_warps<MODE><<<(unsigned)grid, kWThreads, smem, stream>>>(a);
  LV_CUDA(cudaGetLastError());
  if (jgrid > 0) {
    k_jumbo<MODE><<<(unsigned)jgrid, kJBlock, jsmem, stream>>>(a, (int)grid);
    LV_CUDA(cudaGetLastError());
  }
  *ctas = grid + jgrid;
  return ctx ? timing_end(stop, stream) : LV_OK;
}

lv_status ensure_sched(lv_ctx *ctx, int64_t jumbo_cap) {
  if (!ctx->d_ctr && cudaMalloc(&ctx->d_ctr, 2 * sizeof(unsigned long long)) != cudaSuccess) {
    ctx->d_ctr = nullptr;
    return LV_ENOMEM;
  }
  if (jumbo_cap <= ctx->jumbo_cap) return LV_OK;
  LV_CUDA(cudaDeviceSynchronize());
  if (ctx->d_jumbo) cudaFree(ctx->d_jumbo);
  ctx->d_jumbo = nullptr;
  ctx->jumbo_cap = 0;
  const int64_t cap = std::max<int64_t>(jumbo_cap, 1 << 12);
  if (cudaMalloc(&ctx->d_jumbo, sizeof(int64_t) * cap) != cudaSuccess) return LV_ENOMEM;
  ctx->jumbo_cap = cap;
  return LV_OK;
}

// Most batches of more than kJumbo requests that valid offsets allow.
int64_t jumbo_bound(int64_t n_req) { return n_req / (kJumbo + 1) + 1; }

// Partition + warp and jumbo kernels for the given batches.
lv_status run_tiles(lv_ctx *ctx, TileArgs &a, int mode, cudaStream_t stream) {
  ctx->last_grid = 0;
  const int64_t units = a.n_batch + a.n_req;
  // larger tiles fill the per-lane batch groups better and cost fewer tile
  // starts; keep at least six tiles per resident warp for the dynamic
  // schedule's tail (4 kDW measured 3 % faster than 2 kDW on the fit workload)
  const int64_t warps = (int64_t)ctx->sms * (2048 / kWThreads) * kWarps;
  a.D = units / (4 * kDW) >= 6 * warps ? 4 * kDW : units / (2 * kDW) >= 6 * warps ? 2 * kDW : kDW;
  a.n_tiles = (units + a.D - 1) / a.D;
  if (a.n_batch == 0) return LV_OK;
  lv_status st = ensure_tiles(ctx, a.n_tiles + 1);
  if (st != LV_OK) return st;
  st = ensure_sched(ctx, jumbo_bound(a.n_req));
  if (st != LV_OK) return st;
  a.part = ctx->d_tiles;
  a.ctr = ctx->d_ctr;
  a.jumbo_n = ctx->d_ctr + 1;
  a.jumbo = ctx->d_jumbo;
  a.jumbo_cap = ctx->jumbo_cap;
  LV_CUDA(cudaMemsetAsync(ctx->d_ctr, 0, 2 * sizeof(unsigned long long), stream));
  const int64_t nthreads = a.n_batch + 1;
  const int64_t pblocks = std::min<int64_t>((nthreads + 255) / 256, (int64_t)ctx->sms * 16);
  k_partition<<<(unsigned)pblocks, 256, 0, stream>>>(a.off, a.n_batch, a.n_req, a.n_tiles, a.D, ctx->d_tiles,
                                                     ctx->d_status);
  LV_CUDA(cudaGetLastError());
  int64_t *g = &ctx->last_grid;
  const int sms = ctx->sms;
  switch (mode) {
    case M_ATTR: return launch_warps_mode<M_ATTR>(ctx, sms, a, stream, g);
    case M_ATTR | M_FIX: return launch_warps_mode<M_ATTR | M_FIX>(ctx, sms, a, stream, g);
    case M_ATTR | M_TEN: return launch_warps_mode<M_ATTR | M_TEN>(ctx, sms, a, stream, g);
    case M_ATTR | M_TEN | M_FIX: return launch_warps_mode<M_ATTR | M_TEN | M_FIX>(ctx, sms, a, stream, g);
    case M_ATTR | M_F32: return launch_warps_mode<M_ATTR | M_F32>(ctx, sms, a, stream, g);
    case M_ATTR | M_TEN | M_F32: return launch_warps_mode<M_ATTR | M_TEN | M_F32>(ctx, sms, a, stream, g);
    case M_FEAT: return launch_warps_mode<M_FEAT>(ctx, sms, a, stream, g);
    case M_FEAT | M_FIT: return launch_warps_mode<M_FEAT | M_FIT>(ctx, sms, a, stream, g);
    default: return LV_EINVAL;
  }
}

// The one-cluster path for small inputs (k_step); state: the tenant
// accumulator's exact state, or null; L: the totals after the step, or null;
// reset: the state is taken as zero.  The kernel forms every batch constant
// itself, so it reads no K table.
lv_status run_step(lv_ctx *ctx, TileArgs &a, int mode, i128 *state, double *L, int reset, cudaStream_t stream) {
  a.mp.nk = 0;
  a.mp.ktab = nullptr;
  // shared memory: the kernel's fixed part, the tenant table and the received slice entries
  const int slice = (a.H + kStepCtas - 1) / kStepCtas;
  const size_t smem =
      sizeof(StepSmem) + ((mode & M_TEN) ? ten_bytes(a.H) + sizeof(i128) * kStepCtas * (size_t)slice : 0);
  cudaEvent_t stop = nullptr;
  lv_status st = timing_begin(ctx, LV_TIME_TILES, stream, &stop);
  if (st != LV_OK) return st;
  switch (mode) {
    case M_ATTR: k_step<M_ATTR><<<kStepCtas, kStepBlock, smem, stream>>>(a, state, L, reset); break;
    case M_ATTR | M_FIX: k_step<M_ATTR | M_FIX><<<kStepCtas, kStepBlock, smem, stream>>>(a, state, L, reset); break;
    case M_ATTR | M_TEN: k_step<M_ATTR | M_TEN><<<kStepCtas, kStepBlock, smem, stream>>>(a, state, L, reset); break;
    case M_ATTR | M_TEN | M_FIX:
      k_step<M_ATTR | M_TEN | M_FIX><<<kStepCtas, kStepBlock, smem, stream>>>(a, state, L, reset);
      break;
    default: return LV_EINVAL;
  }
  LV_CUDA(cudaGetLastError());
  return timing_end(stop, stream);
}

// Argument checks shared by lv_attribute and lv_attribute_step.
lv_status attr_check(lv_ctx *ctx, const lv_model *model, const lv_batches *b, const double *T, const double *share,
                     const lv_tenant_acc *acc) {
  if (!ctx || check_model(model) != LV_OK) return LV_EINVAL;
  lv_status st = check_batches(b, acc != nullptr);
  if (st != LV_OK) return st;
  if ((T && !aligned(T, 8)) || (share && !aligned(share, 8))) return LV_EINVAL;
  if (acc && (acc->ctx != ctx || acc->n_tenants != b->n_tenants)) return LV_EINVAL;
  return LV_OK;
}

// Launch arguments of an fp64 attribution and its kernel mode.
TileArgs attr_args(lv_ctx *ctx, const lv_batches *b, double *T, double *share, lv_tenant_acc *acc, const ModelP &mp,
                   int *mode) {
  TileArgs a{};
  a.p = b->p;
  a.c = b->c;
  a.ph = b->phase;
  a.ten = acc ? b->tenant : nullptr;
  a.off = b->offsets;
  a.n_req = b->n_req;
  a.n_batch = b->n_batch;
  a.T = T;
  a.share = share;
  a.status = ctx->d_status;
  a.mp = mp;
  *mode = M_ATTR | (mp.fixed ? M_FIX : 0);
  if (acc) {
    *mode |= M_TEN;
    a.ten_pend = acc->d_pend;
    a.n_tenants = acc->n_tenants;
    a.H = std::min<int32_t>(acc->n_tenants, kHotMax);
  }
  return a;
}

// Inputs the one-cluster kernel takes: one serving step.
bool step_sized(const lv_batches *b) {
  return b->n_req <= kSmallMaxReq && b->n_batch <= kSmallMaxBatch && b->n_batch > 0;
}

lv_status fold_tenants(lv_ctx *ctx, lv_tenant_acc *acc, cudaStream_t stream) {
  const int n = acc->n_tenants;
  k_tenant_fold<<<(n + 255) / 256, 256, 0, stream>>>(acc->d_pend, acc->d_state, n, ctx->d_status);
  LV_CUDA(cudaGetLastError());
  return LV_OK;
}

// The exact pass of lv_fit and lv_fit_vtc: per-CTA partials of the fit
// statistics, reduced into totals[4 * NE]; *out points at room for the solves'
// outputs (4 * kFitMaxY FitOut).
lv_status fit_pass(lv_ctx *ctx, const lv_batches *b, const double *y, int32_t n_y, const int64_t split[2],
                   cudaStream_t stream, FitAcc **totals_out, FitOut **out_out) {
  lv_status st = check_batches(b, false);
  if (st != LV_OK) return st;
  if (b->n_batch > 0 && (!y || !aligned(y, 8))) return LV_EINVAL;
  // scratch: per-CTA partials (at most 2048 / kBlock CTAs per SM), totals, solve output
  const int NE = fit_entries(n_y), n_ent = 4 * NE;
  const int64_t max_cta = max_tile_ctas(ctx->sms);
  const size_t o_tot = ((size_t)max_cta * n_ent * sizeof(FitAcc) + 255) & ~(size_t)255;
  const size_t o_out = (o_tot + (size_t)n_ent * sizeof(FitAcc) + 255) & ~(size_t)255;
  const size_t need = o_out + sizeof(FitOut) * 4 * kFitMaxY;
  if (need > ctx->fit_cap) {
    LV_CUDA(cudaDeviceSynchronize());
    if (ctx->d_fit) cudaFree(ctx->d_fit);
    ctx->d_fit = nullptr;
    ctx->fit_cap = 0;
    if (cudaMalloc(&ctx->d_fit, need) != cudaSuccess) return LV_ENOMEM;
    ctx->fit_cap = need;
  }
  unsigned char *base = static_cast<unsigned char *>(ctx->d_fit);
  FitAcc *partial = reinterpret_cast<FitAcc *>(base);
  FitAcc *totals = reinterpret_cast<FitAcc *>(base + o_tot);
  FitOut *out = reinterpret_cast<FitOut *>(base + o_out);

  TileArgs a{};
  a.p = b->p;
  a.c = b->c;
  a.ph = b->phase;
  a.off = b->offsets;
  a.n_req = b->n_req;
  a.n_batch = b->n_batch;
  a.status = ctx->d_status;
  a.mp.split[0] = split[0];
  a.mp.split[1] = split[1];
  a.fit.y = y;
  a.fit.n_y = n_y;
  a.fit.partial = partial;
  ctx->last_grid = 0;
  st = run_tiles(ctx, a, M_FEAT | M_FIT, stream);
  if (st != LV_OK) return st;
  const int n_cta = (int)ctx->last_grid;
  k_fit_reduce<<<n_ent, kFitRedThreads, 0, stream>>>(partial, n_cta, n_ent, totals);
  LV_CUDA(cudaGetLastError());
  *totals_out = totals;
  *out_out = out;
  return LV_OK;
}

// Reads and clears the sticky status after a synchronous fit (syncs `stream`).
lv_status fit_status(lv_ctx *ctx, cudaStream_t stream) {
  int hs = 0;
  LV_CUDA(cudaMemcpyAsync(&hs, ctx->d_status, sizeof(int), cudaMemcpyDeviceToHost, stream));
  LV_CUDA(cudaMemsetAsync(ctx->d_status, 0, sizeof(int), stream));
  LV_CUDA(cudaStreamSynchronize(stream));
  if (hs & kStatusData) return LV_EDATA;
  if (hs & kStatusOverflow) return LV_EOVERFLOW;
  return LV_OK;
}

// lv_whatif and lv_whatif_admit (adm.admit null for the former).
lv_status whatif_run(lv_ctx *ctx, const lv_model *model, const lv_batches *cand, const int32_t *p_new,
                     const int32_t *c_new, const int32_t *phase_new, int64_t n_pending, double *T_new,
                     double *share_new, const AdmitArgs &adm, void *stream_) {
  if (!ctx || check_model(model) != LV_OK || n_pending < 0) return LV_EINVAL;
  lv_status st = check_batches(cand, false);
  if (st != LV_OK) return st;
  if (n_pending > 0 && (!p_new || !c_new || !phase_new || !aligned(p_new, 4) || !aligned(c_new, 4) ||
                        !aligned(phase_new, 4)))
    return LV_EINVAL;
  if ((T_new && !aligned(T_new, 8)) || (share_new && !aligned(share_new, 8))) return LV_EINVAL;
  const int64_t nc = cand->n_batch, np = n_pending;
  if (nc == 0 || np == 0 || (!T_new && !share_new && !adm.admit)) return LV_OK;
  cudaStream_t stream = (cudaStream_t)stream_;
  ModelP mp;
  st = prepare_model(ctx, model, stream, &mp);
  if (st != LV_OK) return st;
  // scratch: candidate sums, segment codes, candidate and pending tables
  const size_t o_feat = 0;
  const size_t o_seg = o_feat + sizeof(int64_t) * 5 * (size_t)nc;
  const size_t o_cand = (o_seg + (size_t)nc + 255) & ~(size_t)255;
  const size_t o_pend = (o_cand + sizeof(CandP) * (size_t)nc + 255) & ~(size_t)255;
  const size_t need = o_pend + sizeof(PendP) * (size_t)np;
  if (need > ctx->wi_cap) {
    LV_CUDA(cudaDeviceSynchronize());
    if (ctx->d_wi) cudaFree(ctx->d_wi);
    ctx->d_wi = nullptr;
    ctx->wi_cap = 0;
    if (cudaMalloc(&ctx->d_wi, need) != cudaSuccess) return LV_ENOMEM;
    ctx->wi_cap = need;
  }
  unsigned char *base = static_cast<unsigned char *>(ctx->d_wi);
  int64_t *bfeat = reinterpret_cast<int64_t *>(base + o_feat);
  uint8_t *bseg = base + o_seg;
  CandP *candp = reinterpret_cast<CandP *>(base + o_cand);
  PendP *pendp = reinterpret_cast<PendP *>(base + o_pend);

  TileArgs a{};
  a.p = cand->p;
  a.c = cand->c;
  a.ph = cand->phase;
  a.off = cand->offsets;
  a.n_req = cand->n_req;
  a.n_batch = nc;
  a.bfeat = bfeat;
  a.bseg = bseg;
  a.status = ctx->d_status;
  a.mp = mp;
  st = run_tiles(ctx, a, M_FEAT, stream);
  if (st != LV_OK) return st;
  k_wi_cand<<<(unsigned)((nc + 127) / 128), 128, 0, stream>>>(mp, bfeat, bseg, nc, candp);
  LV_CUDA(cudaGetLastError());
  k_wi_pend<<<(unsigned)((np + 127) / 128), 128, 0, stream>>>(mp, p_new, c_new, phase_new, np, pendp, adm,
                                                              ctx->d_status);
  LV_CUDA(cudaGetLastError());
  const int64_t gx = (nc + kWiCols - 1) / kWiCols;
  const int64_t rows_per_launch = (int64_t)65535 * kWiRows;
  for (int64_t j = 0; j < np; j += rows_per_launch) {
    const int64_t rows = std::min<int64_t>(rows_per_launch, np - j);
    const dim3 grid((unsigned)gx, (unsigned)((rows + kWiRows - 1) / kWiRows));
    cudaEvent_t stop;
    st = timing_begin(ctx, LV_TIME_PAIRS, stream, &stop);
    if (st != LV_OK) return st;
    k_wi_pairs<<<grid, kWiCols, 0, stream>>>(mp, candp, pendp, nc, np, j, T_new, share_new, adm.slo, adm.admit);
    LV_CUDA(cudaGetLastError());
    st = timing_end(stop, stream);
    if (st != LV_OK) return st;
  }
  st = record_event(ctx->ev_used, stream);
  if (st != LV_OK) return st;
  return LV_OK;
}

}  // namespace

extern "C" {

const char *lv_status_string(lv_status s) {
  switch (s) {
    case LV_OK: return "ok";
    case LV_EINVAL: return "invalid argument";
    case LV_EOVERFLOW: return "int64 overflow";
    case LV_ENODATA: return "not enough data";
    case LV_ESINGULAR: return "singular normal equations";
    case LV_ECUDA: return "CUDA error";
    case LV_EDATA: return "invalid input data";
    case LV_ENOMEM: return "out of device memory";
    case LV_ETIMEOUT: return "a device-side barrier wait timed out";
    default: return "unknown status";
  }
}

lv_status lv_arch_constants(const lv_arch *arch, int64_t phi[3], int64_t *weight_bytes) {
  if (!arch || !phi || !weight_bytes) return LV_EINVAL;
  const int64_t L = arch->n_layers, d = arch->d_model, hq = arch->n_q_heads, hkv = arch->n_kv_heads;
  const int64_t hd = arch->head_dim, F = arch->ffn_dim, wb = arch->weight_bytes, kvb = arch->kv_bytes,
                tp = arch->tp;
  if (L <= 0 || d <= 0 || hq <= 0 || hkv <= 0 || hd <= 0 || F <= 0 || wb <= 0 || kvb <= 0 || tp <= 0)
    return LV_EINVAL;
  if (hq % tp || hkv % tp || F % tp) return LV_EINVAL;
  bool o = false;
  auto mul = [&o](int64_t x, int64_t y) {
    long long r;
    o |= __builtin_mul_overflow((long long)x, (long long)y, &r);
    return (int64_t)r;
  };
  auto add = [&o](int64_t x, int64_t y) {
    long long r;
    o |= __builtin_add_overflow((long long)x, (long long)y, &r);
    return (int64_t)r;
  };
  const int64_t qw = mul(hq, hd), kvw = mul(hkv, hd);
  int64_t P = add(add(add(mul(d, qw), mul(mul(2, d), kvw)), mul(qw, d)), mul(mul(3, d), F));
  const int64_t phi0 = mul(mul(2, L), P) / tp;
  const int64_t phi1 = mul(mul(mul(2, L), kvw), kvb) / tp;
  const int64_t phi2 = mul(mul(2, L), qw) / tp;
  const int64_t W = mul(mul(L, P), wb) / tp;
  if (o) return LV_EOVERFLOW;
  phi[0] = phi0;
  phi[1] = phi1;
  phi[2] = phi2;
  *weight_bytes = W;
  return LV_OK;
}

lv_status lv_ctx_create(lv_ctx **out) {
  if (!out) return LV_EINVAL;
  *out = nullptr;
  lv_ctx *ctx = new (std::nothrow) lv_ctx();
  if (!ctx) return LV_ENOMEM;
  if (cudaGetDevice(&ctx->device) != cudaSuccess ||
      cudaDeviceGetAttribute(&ctx->sms, cudaDevAttrMultiProcessorCount, ctx->device) != cudaSuccess) {
    delete ctx;
    return LV_ECUDA;
  }
  if (cudaMalloc(&ctx->d_status, sizeof(int)) != cudaSuccess) {
    delete ctx;
    return LV_ENOMEM;
  }
  if (cudaMemset(ctx->d_status, 0, sizeof(int)) != cudaSuccess ||
      cudaEventCreateWithFlags(&ctx->ev_built, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&ctx->ev_used, cudaEventDisableTiming) != cudaSuccess) {
    lv_ctx_destroy(ctx);
    return LV_ECUDA;
  }
  *out = ctx;
  return LV_OK;
}

void lv_ctx_destroy(lv_ctx *ctx) {
  if (!ctx) return;
  cudaDeviceSynchronize();
  if (ctx->d_status) cudaFree(ctx->d_status);
  if (ctx->d_tiles) cudaFree(ctx->d_tiles);
  if (ctx->d_ctr) cudaFree(ctx->d_ctr);
  if (ctx->d_jumbo) cudaFree(ctx->d_jumbo);
  if (ctx->d_ktab) cudaFree(ctx->d_ktab);
  if (ctx->d_fit) cudaFree(ctx->d_fit);
  if (ctx->d_wi) cudaFree(ctx->d_wi);
  if (ctx->d_acc) cudaFree(ctx->d_acc);
  if (ctx->h_acc) cudaFreeHost(ctx->h_acc);
  if (ctx->d_probe) cudaFree(ctx->d_probe);
  if (ctx->ev_built) cudaEventDestroy(ctx->ev_built);
  if (ctx->ev_used) cudaEventDestroy(ctx->ev_used);
  for (cudaEvent_t e : ctx->tev) cudaEventDestroy(e);
  delete ctx;
}

lv_status lv_ctx_set_arith(lv_ctx *ctx, int32_t mode) {
  if (!ctx || (mode != LV_ARITH_AUTO && mode != LV_ARITH_FP64)) return LV_EINVAL;
  ctx->arith = mode;
  return LV_OK;
}

lv_status lv_ctx_set_timing(lv_ctx *ctx, int32_t enable) {
  if (!ctx) return LV_EINVAL;
  if (enable & ~(LV_TIME_TILES | LV_TIME_PAIRS)) return LV_EINVAL;
  ctx->timing = enable;
  return LV_OK;
}

lv_status lv_ctx_kernel_time(lv_ctx *ctx, double *ms, int64_t *launches) {
  if (!ctx || !ms || !launches) return LV_EINVAL;
  double tot = 0;
  for (size_t k = 0; k + 1 < ctx->tev_used; k += 2) {
    LV_CUDA(cudaEventSynchronize(ctx->tev[k + 1]));
    float m = 0;
    LV_CUDA(cudaEventElapsedTime(&m, ctx->tev[k], ctx->tev[k + 1]));
    tot += m;
  }
  *ms = tot;
  *launches = (int64_t)(ctx->tev_used / 2);
  ctx->tev_used = 0;
  return LV_OK;
}

lv_status lv_ctx_status(lv_ctx *ctx, void *stream) {
  if (!ctx) return LV_EINVAL;
  LV_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
  int h = 0;
  LV_CUDA(cudaMemcpy(&h, ctx->d_status, sizeof(int), cudaMemcpyDeviceToHost));
  LV_CUDA(cudaMemset(ctx->d_status, 0, sizeof(int)));
  if (h & kStatusTimeout) return LV_ETIMEOUT;
  if (h & kStatusData) return LV_EDATA;
  return LV_OK;
}

lv_status lv_features(lv_ctx *ctx, const lv_arch *arch, const lv_model *model, const lv_batches *b,
                      int64_t *req_feat, int64_t *batch_feat, uint8_t *batch_seg, void *stream_) {
  if (!ctx) return LV_EINVAL;
  lv_status st = check_batches(b, false);
  if (st != LV_OK) return st;
  if (req_feat && (!arch || !aligned(req_feat, 8))) return LV_EINVAL;
  if (batch_seg && check_model(model) != LV_OK) return LV_EINVAL;
  if (batch_feat && !aligned(batch_feat, 8)) return LV_EINVAL;
  cudaStream_t stream = (cudaStream_t)stream_;
  if (req_feat) {
    int64_t phi[3], W;
    st = lv_arch_constants(arch, phi, &W);
    if (st != LV_OK) return st;
    if (b->n_req > 0) {
      const int64_t blocks = std::min<int64_t>((b->n_req + 255) / 256, (int64_t)ctx->sms * 8);
      k_req_features<<<(unsigned)blocks, 256, 0, stream>>>(b->p, b->c, b->n_req, phi[0], phi[1], phi[2], req_feat,
                                                           ctx->d_status);
      LV_CUDA(cudaGetLastError());
    }
  }
  if (batch_feat || batch_seg) {
    TileArgs a{};
    a.p = b->p;
    a.c = b->c;
    a.ph = b->phase;
    a.off = b->offsets;
    a.n_req = b->n_req;
    a.n_batch = b->n_batch;
    a.bfeat = batch_feat;
    a.bseg = batch_seg;
    a.status = ctx->d_status;
    if (model) {
      a.mp.split[0] = model->split[0];
      a.mp.split[1] = model->split[1];
    }
    st = run_tiles(ctx, a, M_FEAT, stream);
    if (st != LV_OK) return st;
  }
  return LV_OK;
}

lv_status lv_batch_latency(lv_ctx *ctx, const lv_model *model, const int64_t *batch_feat, const uint8_t *batch_seg,
                           int64_t n_batch, double *T, void *stream_) {
  if (!ctx || check_model(model) != LV_OK || n_batch < 0) return LV_EINVAL;
  if (n_batch > 0 && (!batch_feat || !batch_seg || !T || !aligned(batch_feat, 8) || !aligned(T, 8)))
    return LV_EINVAL;
  if (n_batch == 0) return LV_OK;
  cudaStream_t stream = (cudaStream_t)stream_;
  ModelP mp;
  lv_status st = prepare_model(ctx, model, stream, &mp);
  if (st != LV_OK) return st;
  const int64_t blocks = std::min<int64_t>((n_batch + 255) / 256, (int64_t)ctx->sms * 8);
  if (mp.fixed)
    k_batch_latency<true><<<(unsigned)blocks, 256, 0, stream>>>(mp, batch_feat, batch_seg, n_batch, T,
                                                                ctx->d_status);
  else
    k_batch_latency<false><<<(unsigned)blocks, 256, 0, stream>>>(mp, batch_feat, batch_seg, n_batch, T,
                                                                 ctx->d_status);
  LV_CUDA(cudaGetLastError());
  st = record_event(ctx->ev_used, stream);
  if (st != LV_OK) return st;
  return LV_OK;
}

lv_status lv_attribute(lv_ctx *ctx, const lv_model *model, const lv_batches *b, double *T, double *share,
                       lv_tenant_acc *acc, void *stream_) {
  lv_status st = attr_check(ctx, model, b, T, share, acc);
  if (st != LV_OK) return st;
  if (b->n_batch > 0 && !T && !share && !acc) return LV_OK;
  cudaStream_t stream = (cudaStream_t)stream_;
  ModelP mp;
  int mode = 0;
  if (step_sized(b)) {
    // one serving step: a single cluster, no partition, scheduling counters or K table
    model_params(ctx, model, &mp);
    TileArgs a = attr_args(ctx, b, T, share, acc, mp, &mode);
    st = run_step(ctx, a, mode, acc ? acc->d_state : nullptr, nullptr, 0, stream);
    if (st != LV_OK) return st;
    if (acc && acc->n_tenants > kHotMax) return fold_tenants(ctx, acc, stream);
    return LV_OK;
  }
  st = prepare_model(ctx, model, stream, &mp);
  if (st != LV_OK) return st;
  TileArgs a = attr_args(ctx, b, T, share, acc, mp, &mode);
  st = run_tiles(ctx, a, mode, stream);
  if (st != LV_OK) return st;
  st = record_event(ctx->ev_used, stream);
  if (st != LV_OK) return st;
  if (acc) return fold_tenants(ctx, acc, stream);
  return LV_OK;
}

lv_status lv_attribute_step(lv_ctx *ctx, const lv_model *model, const lv_batches *b, double *T, double *share,
                            lv_tenant_acc *acc, double *L, int32_t flags, void *stream_) {
  if ((flags & ~LV_STEP_RESET) != 0 || (!acc && (L || (flags & LV_STEP_RESET))) || (L && !aligned(L, 8)))
    return LV_EINVAL;
  lv_status st = attr_check(ctx, model, b, T, share, acc);
  if (st != LV_OK) return st;
  const int reset = (flags & LV_STEP_RESET) ? 1 : 0;
  if (step_sized(b) && (!acc || acc->n_tenants <= kHotMax)) {
    if (!T && !share && !acc) return LV_OK;
    // the whole step in one launch: attribution, tenant add and totals
    ModelP mp;
    model_params(ctx, model, &mp);
    int mode = 0;
    TileArgs a = attr_args(ctx, b, T, share, acc, mp, &mode);
    return run_step(ctx, a, mode, acc ? acc->d_state : nullptr, L, reset, (cudaStream_t)stream_);
  }
  if (reset) {
    st = lv_tenant_acc_reset(acc, stream_);
    if (st != LV_OK) return st;
  }
  st = lv_attribute(ctx, model, b, T, share, acc, stream_);
  if (st != LV_OK) return st;
  return L ? lv_tenant_totals(ctx, acc, L, stream_) : LV_OK;
}

lv_status lv_attribute_f32(lv_ctx *ctx, const lv_model *model, const lv_batches *b, float *T, float *share,
                           lv_tenant_acc *acc, void *stream_) {
  if (!ctx || check_model(model) != LV_OK) return LV_EINVAL;
  lv_status st = check_batches(b, acc != nullptr);
  if (st != LV_OK) return st;
  if ((T && !aligned(T, 4)) || (share && !aligned(share, 4))) return LV_EINVAL;
  if (acc && (acc->ctx != ctx || acc->n_tenants != b->n_tenants)) return LV_EINVAL;
  if (!T && !share && !acc) return LV_OK;
  cudaStream_t stream = (cudaStream_t)stream_;
  ModelP mp;
  st = prepare_model(ctx, model, stream, &mp);
  if (st != LV_OK) return st;
  TileArgs a{};
  a.p = b->p;
  a.c = b->c;
  a.ph = b->phase;
  a.ten = acc ? b->tenant : nullptr;
  a.off = b->offsets;
  a.n_req = b->n_req;
  a.n_batch = b->n_batch;
  a.T32 = T;
  a.share32 = share;
  a.status = ctx->d_status;
  a.mp = mp;
  int mode = M_ATTR | M_F32;
  if (acc) {
    mode |= M_TEN;
    a.ten_pend = acc->d_pend;
    a.n_tenants = acc->n_tenants;
    a.H = std::min<int32_t>(acc->n_tenants, kHotMax);
  }
  st = run_tiles(ctx, a, mode, stream);
  if (st != LV_OK) return st;
  st = record_event(ctx->ev_used, stream);
  if (st != LV_OK) return st;
  if (acc) return fold_tenants(ctx, acc, stream);
  return LV_OK;
}

lv_status lv_tenant_acc_create(lv_ctx *ctx, int32_t n_tenants, lv_tenant_acc **out) {
  if (!ctx || !out || n_tenants <= 0) return LV_EINVAL;
  *out = nullptr;
  lv_tenant_acc *acc = new (std::nothrow) lv_tenant_acc();
  if (!acc) return LV_ENOMEM;
  acc->ctx = ctx;
  acc->n_tenants = n_tenants;
  if (cudaMalloc(&acc->d_pend, sizeof(unsigned long long) * 4 * (size_t)n_tenants) != cudaSuccess ||
      cudaMalloc(&acc->d_state, sizeof(i128) * (size_t)n_tenants) != cudaSuccess) {
    lv_tenant_acc_destroy(acc);
    return LV_ENOMEM;
  }
  if (cudaMemset(acc->d_pend, 0, sizeof(unsigned long long) * 4 * (size_t)n_tenants) != cudaSuccess ||
      cudaMemset(acc->d_state, 0, sizeof(i128) * (size_t)n_tenants) != cudaSuccess ||
      cudaDeviceSynchronize() != cudaSuccess) {
    lv_tenant_acc_destroy(acc);
    return LV_ECUDA;
  }
  *out = acc;
  return LV_OK;
}

void lv_tenant_acc_destroy(lv_tenant_acc *acc) {
  if (!acc) return;
  cudaDeviceSynchronize();
  if (acc->d_pend) cudaFree(acc->d_pend);
  if (acc->d_state) cudaFree(acc->d_state);
  delete acc;
}

lv_status lv_tenant_acc_reset(lv_tenant_acc *acc, void *stream) {
  if (!acc) return LV_EINVAL;
  LV_CUDA(cudaMemsetAsync(acc->d_pend, 0, sizeof(unsigned long long) * 4 * (size_t)acc->n_tenants,
                          (cudaStream_t)stream));
  LV_CUDA(cudaMemsetAsync(acc->d_state, 0, sizeof(i128) * (size_t)acc->n_tenants, (cudaStream_t)stream));
  return LV_OK;
}

lv_status lv_tenant_accumulate(lv_ctx *ctx, lv_tenant_acc *acc, const double *share, const int32_t *tenant,
                               int64_t n_req, void *stream_) {
  if (!ctx || !acc || acc->ctx != ctx || n_req < 0) return LV_EINVAL;
  if (n_req > 0 && (!share || !tenant || !aligned(share, 8) || !aligned(tenant, 4))) return LV_EINVAL;
  cudaStream_t stream = (cudaStream_t)stream_;
  if (n_req > 0) {
    const int H = std::min<int32_t>(acc->n_tenants, kHotMax);
    const size_t smem = ten_bytes(H);
    static bool configured = false;
    if (!configured) {
      LV_CUDA(cudaFuncSetAttribute(k_tenant_acc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   (int)ten_bytes(kHotMax)));
      configured = true;
    }
    const int64_t blocks = std::min<int64_t>((n_req + kBlock - 1) / kBlock, (int64_t)ctx->sms * 4);
    k_tenant_acc<<<(unsigned)blocks, kBlock, smem, stream>>>(share, tenant, n_req, acc->d_pend, acc->n_tenants, H,
                                                              ctx->d_status);
    LV_CUDA(cudaGetLastError());
  }
  return fold_tenants(ctx, acc, stream);
}

lv_status lv_tenant_totals(lv_ctx *ctx, lv_tenant_acc *acc, double *L, void *stream_) {
  if (!ctx || !acc || acc->ctx != ctx || !L || !aligned(L, 8)) return LV_EINVAL;
  const int n = acc->n_tenants;
  k_tenant_totals<<<(n + 255) / 256, 256, 0, (cudaStream_t)stream_>>>(acc->d_state, L, n);
  LV_CUDA(cudaGetLastError());
  return LV_OK;
}

int64_t lv_tenant_acc_state_bytes(const lv_tenant_acc *acc) {
  return acc ? (int64_t)sizeof(i128) * acc->n_tenants : 0;
}

lv_status lv_tenant_acc_export(lv_tenant_acc *acc, void *host_state, int64_t bytes, void *stream) {
  if (!acc || !host_state || bytes != lv_tenant_acc_state_bytes(acc)) return LV_EINVAL;
  LV_CUDA(cudaMemcpyAsync(host_state, acc->d_state, (size_t)bytes, cudaMemcpyDeviceToHost, (cudaStream_t)stream));
  LV_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
  return LV_OK;
}

lv_status lv_tenant_acc_import(lv_tenant_acc *acc, const void *host_state, int64_t bytes, void *stream) {
  if (!acc || !host_state || bytes != lv_tenant_acc_state_bytes(acc)) return LV_EINVAL;
  LV_CUDA(cudaMemsetAsync(acc->d_pend, 0, sizeof(unsigned long long) * 4 * (size_t)acc->n_tenants,
                          (cudaStream_t)stream));
  LV_CUDA(cudaMemcpyAsync(acc->d_state, host_state, (size_t)bytes, cudaMemcpyHostToDevice, (cudaStream_t)stream));
  LV_CUDA(cudaStreamSynchronize((cudaStream_t)stream));
  return LV_OK;
}

}  // extern "C"

extern "C" {

lv_status lv_fit(lv_ctx *ctx, const lv_batches *b, const double *y, int32_t n_y, lv_model *inout,
                 lv_fit_report *rep, void *stream_) {
  if (!ctx || !inout || n_y < 1 || n_y > kFitMaxY) return LV_EINVAL;
  for (int k = 1; k < n_y; ++k)
    if (inout[k].split[0] != inout[0].split[0] || inout[k].split[1] != inout[0].split[1]) return LV_EINVAL;
  cudaStream_t stream = (cudaStream_t)stream_;
  FitAcc *totals = nullptr;
  FitOut *out = nullptr;
  lv_status st = fit_pass(ctx, b, y, n_y, inout[0].split, stream, &totals, &out);
  if (st != LV_OK) return st;
  k_fit_solve<<<4 * kFitMaxY, 32, 0, stream>>>(totals, n_y, out);
  LV_CUDA(cudaGetLastError());
  FitOut h[4 * kFitMaxY];
  LV_CUDA(cudaMemcpyAsync(h, out, sizeof(FitOut) * 4 * (size_t)n_y, cudaMemcpyDeviceToHost, stream));
  st = fit_status(ctx, stream);
  if (st != LV_OK) return st;
  for (int k = 0; k < n_y; ++k) {
    for (int g = 0; g < 4; ++g) {
      const FitOut &o = h[k * 4 + g];
      if (rep) {
        rep[k].n[g] = o.n;
        rep[k].status[g] = o.status;
        rep[k].dropped[g] = o.dropped;
        rep[k].ssr[g] = o.ssr;
        rep[k].r2[g] = o.r2;
      }
      if (o.status == LV_OK) {
        lv_coef &c = inout[k].seg[g >> 1][g & 1];
        c.beta = o.coef[0];
        c.a1 = o.coef[1];
        c.a2 = o.coef[2];
        c.a3 = o.coef[3];
        c.a4 = o.coef[4];
      }
    }
  }
  return LV_OK;
}

lv_status lv_fit_vtc(lv_ctx *ctx, const lv_batches *b, const double *y, int32_t n_y, double *coef, int32_t *status,
                     int64_t *count, void *stream_) {
  if (!ctx || !coef || !status || n_y < 1 || n_y > kFitMaxY) return LV_EINVAL;
  cudaStream_t stream = (cudaStream_t)stream_;
  FitAcc *totals = nullptr;
  FitOut *out = nullptr;
  const int64_t split[2] = {0, 0};  // the groups do not matter: the line pools all four
  lv_status st = fit_pass(ctx, b, y, n_y, split, stream, &totals, &out);
  if (st != LV_OK) return st;
  static_assert(sizeof(VtcOut) * kFitMaxY <= sizeof(FitOut) * 4 * kFitMaxY, "VTC output fits the solve area");
  VtcOut *vo = reinterpret_cast<VtcOut *>(out);
  k_vtc_solve<<<1, 32, 0, stream>>>(totals, n_y, vo);
  LV_CUDA(cudaGetLastError());
  VtcOut h[kFitMaxY];
  LV_CUDA(cudaMemcpyAsync(h, vo, sizeof(VtcOut) * (size_t)n_y, cudaMemcpyDeviceToHost, stream));
  st = fit_status(ctx, stream);
  if (st != LV_OK) return st;
  for (int k = 0; k < n_y; ++k) {
    status[k] = h[k].status;
    if (count) count[k] = h[k].n;
    if (h[k].status == LV_OK) {
      coef[2 * k] = h[k].beta;
      coef[2 * k + 1] = h[k].a;
    }
  }
  return LV_OK;
}

lv_status lv_accuracy(lv_ctx *ctx, const double *y, const double *T, int64_t n, lv_accuracy_report *rep,
                      void *stream_) {
  if (!ctx || !rep || n < 0 || n >= ((int64_t)1 << 32) ||
      (n > 0 && (!y || !T || !aligned(y, 8) || !aligned(T, 8))))
    return LV_EINVAL;
  const double nan = std::nan("");
  rep->n = 0;
  rep->r2_ssr = rep->r2_corr = rep->mean_rel = rep->p50 = rep->p90 = rep->p99 = nan;
  if (n == 0) return LV_OK;
  cudaStream_t stream = (cudaStream_t)stream_;
  if (!ctx->h_acc) {
    void *h = nullptr, *d = nullptr;
    if (cudaHostAlloc(&h, 16 * sizeof(double), cudaHostAllocMapped) != cudaSuccess) return LV_ENOMEM;
    if (cudaHostGetDevicePointer(&d, h, 0) != cudaSuccess) {
      cudaFreeHost(h);
      return LV_ECUDA;
    }
    ctx->h_acc = static_cast<double *>(h);
    ctx->hd_acc = static_cast<double *>(d);
  }
  constexpr size_t acc_dyn = kAccStage * sizeof(uint64_t);
  if (ctx->acc_occ == 0) {
    LV_CUDA(cudaFuncSetAttribute(k_acc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)acc_dyn));
    LV_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&ctx->acc_occ, k_acc, kAccBlock, acc_dyn));
    if (ctx->acc_occ <= 0) return LV_ECUDA;
  }
  // a cooperative launch: at most the blocks that fit at once, each looping over its share
  const int blocks = (int)std::max<int64_t>(
      1, std::min<int64_t>((n + kAccBlock - 1) / kAccBlock, (int64_t)ctx->sms * ctx->acc_occ));
  // a fixed head (barrier, list cursors, results, digit histograms: zeroed
  // once at allocation, and every call leaves the barrier, cursors and
  // histograms at zero), then the relative errors' bit patterns, the
  // candidate lists and the block partials
  constexpr size_t o_bar = 0, o_err = 64, o_lost = 68, o_hist1 = 256, o_hist2 = o_hist1 + 8 * kSelBins,
                   o_rel = 45056;
  static_assert(o_hist2 + 4 * kAccTargets * kSelBins <= o_rel, "accuracy scratch head");
  const size_t rel_bytes = ((size_t)n * sizeof(uint64_t) + 255) & ~(size_t)255;
  const size_t o_sorted = o_rel + rel_bytes, o_bucket = o_sorted + rel_bytes;
  const size_t o_segs = o_bucket + sizeof(uint64_t) * kAccTargets * kSelBins * kAccBucket;
  const size_t o_part = o_segs + ((sizeof(uint64_t) * 2 * kAccTargets * (size_t)blocks + 255) & ~(size_t)255);
  const size_t need = o_part + sizeof(uint64_t) * kAccPartW * (size_t)blocks;
  if (need > ctx->acc_cap) {
    LV_CUDA(cudaDeviceSynchronize());
    if (ctx->d_acc) cudaFree(ctx->d_acc);
    ctx->d_acc = nullptr;
    ctx->acc_cap = 0;
    if (cudaMalloc(&ctx->d_acc, need) != cudaSuccess) return LV_ENOMEM;
    if (cudaMemset(ctx->d_acc, 0, o_rel) != cudaSuccess) return LV_ECUDA;
    ctx->acc_cap = need;
  }
  unsigned char *base = static_cast<unsigned char *>(ctx->d_acc);
  AccArgs a;
  a.y = y;
  a.T = T;
  a.n = n;
  a.relbits = reinterpret_cast<uint64_t *>(base + o_rel);
  a.cand = reinterpret_cast<uint64_t *>(base + o_sorted);
  a.bucket = reinterpret_cast<uint64_t *>(base + o_bucket);
  a.segs = reinterpret_cast<uint64_t *>(base + o_segs);
  a.part = reinterpret_cast<uint64_t *>(base + o_part);
  a.res = ctx->hd_acc;
  a.err = reinterpret_cast<int *>(base + o_err);
  a.lost = reinterpret_cast<int *>(base + o_lost);
  a.hist1 = reinterpret_cast<unsigned int *>(base + o_hist1);
  a.hist2 = reinterpret_cast<unsigned int *>(base + o_hist2);
  a.bar = reinterpret_cast<unsigned int *>(base + o_bar);
  volatile double *h = ctx->h_acc;  // eight sums, three percentile bit patterns, error word
  *reinterpret_cast<volatile int *>(ctx->h_acc + 11) = 0;
  void *args[] = {&a};
  LV_CUDA(cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(k_acc), dim3(blocks), dim3(kAccBlock), args,
                                      acc_dyn, stream));
  LV_CUDA(cudaStreamSynchronize(stream));
  if (*reinterpret_cast<volatile int *>(ctx->h_acc + 11)) {
    // a block waited out a barrier: reset the barrier and its error word for the next call
    LV_CUDA(cudaMemset(base + o_bar, 0, 8));
    LV_CUDA(cudaMemset(base + o_err, 0, sizeof(int)));
    return LV_ETIMEOUT;
  }
  const double m = h[0];
  rep->n = (int64_t)m;
  if (m == 0) return LV_OK;
  // sxx, syy, sxy, ssr: plain sums (fp64 path) or the same times m 2^(2S)
  // (exact path); both R^2 are ratios, so the common factor cancels
  const double sxx = h[3], syy = h[4], sxy = h[5], ssr = h[6], srel = h[7];
  rep->r2_ssr = sxx != 0 ? 1.0 - ssr / sxx : nan;
  rep->r2_corr = (sxx != 0 && syy != 0) ? sxy * sxy / (sxx * syy) : nan;
  rep->mean_rel = srel / m;
  rep->p50 = h[8];
  rep->p90 = h[9];
  rep->p99 = h[10];
  return LV_OK;
}

lv_status lv_ctx_selftest_barrier(lv_ctx *ctx, void *stream_) {
  if (!ctx) return LV_EINVAL;
  cudaStream_t stream = (cudaStream_t)stream_;
  if (!ctx->d_probe && cudaMalloc(&ctx->d_probe, 16) != cudaSuccess) return LV_ENOMEM;
  LV_CUDA(cudaMemsetAsync(ctx->d_probe, 0, 16, stream));
  unsigned int *bar = static_cast<unsigned int *>(ctx->d_probe);
  int *err = reinterpret_cast<int *>(bar + 2);
  void *args[] = {&bar, &err};
  LV_CUDA(cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(k_barrier_probe), dim3(2), dim3(32), args, 0,
                                      stream));
  int h = 0;
  LV_CUDA(cudaMemcpyAsync(&h, err, sizeof(int), cudaMemcpyDeviceToHost, stream));
  LV_CUDA(cudaStreamSynchronize(stream));
  return h ? LV_ETIMEOUT : LV_OK;
}

lv_status lv_whatif(lv_ctx *ctx, const lv_model *model, const lv_batches *cand, const int32_t *p_new,
                    const int32_t *c_new, const int32_t *phase_new, int64_t n_pending, double *T_new,
                    double *share_new, void *stream_) {
  return whatif_run(ctx, model, cand, p_new, c_new, phase_new, n_pending, T_new, share_new, AdmitArgs{}, stream_);
}

lv_status lv_whatif_admit(lv_ctx *ctx, const lv_model *model, const lv_batches *cand, const int32_t *p_new,
                          const int32_t *c_new, const int32_t *phase_new, const int32_t *tenant_new,
                          int64_t n_pending, const double *L, const double *budget, int32_t n_tenants, double slo,
                          double *T_new, double *share_new, uint8_t *admit, void *stream_) {
  if (!admit || n_tenants <= 0 || (n_pending > 0 && (!tenant_new || !aligned(tenant_new, 4))) || !L || !budget ||
      !aligned(L, 8) || !aligned(budget, 8))
    return LV_EINVAL;
  AdmitArgs adm{tenant_new, L, budget, n_tenants, slo, admit};
  return whatif_run(ctx, model, cand, p_new, c_new, phase_new, n_pending, T_new, share_new, adm, stream_);
}

}  // extern "C"

// ---------------------------------------------------------------- allocation-free attribution
//
// lv_attribute_noalloc: the same kernels as lv_attribute (no tenant pass),
// with the partition and the per-model constant table in a static device array
// instead of a context's cudaMalloc'd scratch.

namespace {

constexpr int64_t kNoAllocMaxTiles = 1 << 16;  // => n_batch + n_req <= 65,536 * kDW
constexpr size_t kNoAllocPartBytes = sizeof(TilePart) * (size_t)(kNoAllocMaxTiles + 1);
constexpr size_t kNoAllocTabOffset = (kNoAllocPartBytes + 255) & ~(size_t)255;
constexpr size_t kNoAllocCtrOffset = (kNoAllocTabOffset + sizeof(KEntry) * 4 * (kKTableN + 1) + 255) & ~(size_t)255;
constexpr size_t kNoAllocJumboOffset = kNoAllocCtrOffset + 256;
constexpr int64_t kNoAllocJumboCap = kNoAllocMaxTiles * kDW / (kJumbo + 1) + 1;
constexpr size_t kNoAllocBytes = kNoAllocJumboOffset + sizeof(int64_t) * (size_t)kNoAllocJumboCap;
// the size stated in include/llmvisor.h ("about 2.6 MB")
static_assert(kNoAllocBytes > 2500000 && kNoAllocBytes < 2700000, "no-alloc scratch size as documented");

}  // namespace

// The scratch itself: one copy per device that loads the library.
static __device__ __align__(256) unsigned char lv_noalloc_scratch[kNoAllocBytes];

namespace {

constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
void *g_noalloc_ptr[kNoAllocMaxDevices] = {};
int g_noalloc_sms[kNoAllocMaxDevices] = {};

// Device address of the scratch array on `dev` (looked up once per device, with
// that device current).
lv_status noalloc_scratch(int dev, void **ptr, int *sms) {
  if (dev < 0 || dev >= kNoAllocMaxDevices) return LV_EINVAL;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, lv_noalloc_scratch) != cudaSuccess || !p) return LV_ECUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return LV_ECUDA;
    g_noalloc_ptr[dev] = p;
    g_noalloc_sms[dev] = n;
  }
  *ptr = g_noalloc_ptr[dev];
  *sms = g_noalloc_sms[dev];
  return LV_OK;
}

}  // namespace

extern "C" lv_status lv_attribute_noalloc(const lv_model *model, const lv_batches *b, double *T, double *share,
                                          int32_t *status, void *stream_) {
  if (check_model(model) != LV_OK) return LV_EINVAL;
  lv_status st = check_batches(b, false);
  if (st != LV_OK) return st;
  if (T && !aligned(T, 8)) return LV_EINVAL;
  if (share && !aligned(share, 8)) return LV_EINVAL;
  if (status && !aligned(status, 4)) return LV_EINVAL;
  const int64_t n_tiles = (b->n_batch + b->n_req + kDW - 1) / kDW;
  if (n_tiles > kNoAllocMaxTiles) return LV_EINVAL;
  int dev = 0;
  LV_CUDA(cudaGetDevice(&dev));
  void *scratch = nullptr;
  int sms = 0;
  st = noalloc_scratch(dev, &scratch, &sms);
  if (st != LV_OK) return st;
  cudaStream_t stream = (cudaStream_t)stream_;
  if (status) LV_CUDA(cudaMemsetAsync(status, 0, sizeof(int32_t), stream));
  if (b->n_batch == 0 || (!T && !share)) return LV_OK;

  ModelP mp;
  std::memset(&mp, 0, sizeof(mp));
  for (int s = 0; s < 4; ++s) {
    const lv_coef &k = model->seg[s >> 1][s & 1];
    mp.coef[s][0] = k.beta;
    mp.coef[s][1] = k.a1;
    mp.coef[s][2] = k.a2;
    mp.coef[s][3] = k.a3;
    mp.coef[s][4] = k.a4;
  }
  mp.split[0] = model->split[0];
  mp.split[1] = model->split[1];
  mp.nk = kKTableN;
  mp.fixed = derive_fixed(model, kKTableN, &mp) ? 1 : 0;
  KEntry *ktab = reinterpret_cast<KEntry *>(static_cast<unsigned char *>(scratch) + kNoAllocTabOffset);
  mp.ktab = ktab;
  const int nk = 4 * (kKTableN + 1);
  k_ktable<<<(nk + 255) / 256, 256, 0, stream>>>(mp, ktab);
  LV_CUDA(cudaGetLastError());

  TileArgs a{};
  a.p = b->p;
  a.c = b->c;
  a.ph = b->phase;
  a.off = b->offsets;
  a.n_req = b->n_req;
  a.n_batch = b->n_batch;
  a.T = T;
  a.share = share;
  a.status = status;
  a.mp = mp;
  a.n_tiles = n_tiles;
  a.D = kDW;
  unsigned char *base = static_cast<unsigned char *>(scratch);
  TilePart *part = reinterpret_cast<TilePart *>(base);
  a.part = part;
  a.ctr = reinterpret_cast<unsigned long long *>(base + kNoAllocCtrOffset);
  a.jumbo_n = a.ctr + 1;
  a.jumbo = reinterpret_cast<int64_t *>(base + kNoAllocJumboOffset);
  a.jumbo_cap = kNoAllocJumboCap;
  LV_CUDA(cudaMemsetAsync(a.ctr, 0, 2 * sizeof(unsigned long long), stream));
  const int64_t pblocks = std::min<int64_t>((b->n_batch + 1 + 255) / 256, (int64_t)sms * 16);
  k_partition<<<(unsigned)pblocks, 256, 0, stream>>>(a.off, a.n_batch, a.n_req, a.n_tiles, kDW, part, status);
  LV_CUDA(cudaGetLastError());
  int64_t ctas = 0;
  return mp.fixed ? launch_warps_mode<M_ATTR | M_FIX>(nullptr, sms, a, stream, &ctas)
                  : launch_warps_mode<M_ATTR>(nullptr, sms, a, stream, &ctas);
}
