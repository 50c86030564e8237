"""Seeded synthetic inputs for the attribution path.

This module only draws random inputs: request records (new tokens ``p``, context
``c``, phase, tenant), CSR batch offsets, model-architecture integers and the
coefficient sets handed to the latency model.  It evaluates nothing of the
method itself (no features, no Eq. 1, no shares, no fit), so both the CPU oracle
and the CUDA path can consume the very same arrays.

Shapes follow the paper's workloads: Llama3.1-8B and Qwen2.5-14B/32B served with
tensor parallelism, prefill and decode steps, 128-2048 concurrent requests with
heavy-tailed lengths (Section 3.1, Appendix A).  The paper's vLLM traces are not
available; these recipes stand in for them.

Conventions for every generated workload (all numpy arrays):

* ``p, c, phase, tenant``: int32[n_req], struct-of-arrays.  ``phase`` is 1 for a
  prefill request and 0 for a decode request; decode requests have ``p == 1``.
* ``offsets``: int64[n_batch + 1], ``offsets[0] == 0``, ``offsets[-1] == n_req``.
* ``coef``: float64[4, 5] indexed ``[phase * 2 + regime]`` with columns
  ``(beta, a1, a2, a3, a4)``; regime 0 is memory-bound, 1 compute-bound.
* ``split``: int64[2], the per-phase threshold on the batch's total new tokens.
"""

from __future__ import annotations

import dataclasses
import math

import numpy as np

__all__ = [
    "ARCHS", "Workload", "WhatIf", "config", "whatif_config", "step_config", "random_batches",
    "draw_coefficients", "zipf_tenants", "SEED_BASE",
]

SEED_BASE = 20260382

# Architecture integers: (n_layers, d_model, n_q_heads, n_kv_heads, head_dim,
# ffn_dim, weight_bytes, kv_bytes, tp).  Public model shapes.
ARCHS = {
    "llama3.1-8b": (32, 4096, 32, 8, 128, 14336, 2, 2, 1),
    "qwen2.5-14b": (48, 5120, 40, 8, 128, 13824, 2, 2, 2),
    "qwen2.5-32b": (64, 5120, 40, 8, 128, 27648, 2, 2, 4),
}

# Per-model cost scales used only to draw plausible coefficient magnitudes:
# weight bytes per step, FLOPs per new token, KV bytes per context token and
# attention FLOPs per squared new token for the shapes above (hand-computed
# dense-transformer counts with a gated FFN).  Any value would do for parity,
# since both sides receive the drawn coefficients as inputs.
_COST_SCALES = {
    "llama3.1-8b": (13_958_643_712, 13_958_643_712, 131_072, 262_144),
    "qwen2.5-14b": (13_212_057_600, 13_212_057_600, 98_304, 245_760),
    "qwen2.5-32b": (15_602_810_880, 15_602_810_880, 65_536, 163_840),
}
_BW = 8.0e12   # modelled HBM bytes/s
_PK = 1.88e15  # modelled dense FLOP/s


@dataclasses.dataclass
class Workload:
    name: str
    arch: np.ndarray          # int32[9]
    p: np.ndarray             # int32[n_req]
    c: np.ndarray             # int32[n_req]
    phase: np.ndarray         # int32[n_req]
    tenant: np.ndarray        # int32[n_req]
    offsets: np.ndarray       # int64[n_batch+1]
    n_tenants: int
    coef: np.ndarray          # float64[4,5]
    split: np.ndarray         # int64[2]
    noise: np.ndarray | None = None   # float64[n_batch], multiplicative latency noise (fit workload)
    seed: int = 0

    @property
    def n_req(self) -> int:
        return int(self.p.shape[0])

    @property
    def n_batch(self) -> int:
        return int(self.offsets.shape[0] - 1)


@dataclasses.dataclass
class WhatIf:
    name: str
    arch: np.ndarray
    cand: Workload            # candidate batches (tenant unused)
    p_new: np.ndarray         # int32[n_pending]
    c_new: np.ndarray
    phase_new: np.ndarray
    coef: np.ndarray
    split: np.ndarray
    seed: int = 0

    @property
    def n_pending(self) -> int:
        return int(self.p_new.shape[0])


def _offsets_from_sizes(sizes: np.ndarray) -> np.ndarray:
    off = np.zeros(sizes.shape[0] + 1, dtype=np.int64)
    np.cumsum(sizes, out=off[1:])
    return off


def _log_uniform_int(rng, n, hi):
    """floor(exp(U(0, ln hi))) clipped to [1, hi]."""
    v = np.floor(np.exp(rng.uniform(0.0, math.log(hi), size=n)))
    return np.clip(v, 1, hi).astype(np.int32)


def _lognormal_int(rng, n, mu, sigma, lo, hi):
    v = np.rint(rng.lognormal(mean=mu, sigma=sigma, size=n))
    return np.clip(v, lo, hi).astype(np.int32)


def zipf_tenants(rng, n, n_tenants, s):
    """Tenant ids with P(id = k-1) proportional to k^-s, k = 1..n_tenants."""
    w = np.arange(1, n_tenants + 1, dtype=np.float64) ** (-s)
    cdf = np.cumsum(w)
    cdf /= cdf[-1]
    u = rng.random(n)
    t = np.searchsorted(cdf, u, side="right")
    return np.minimum(t, n_tenants - 1).astype(np.int32)


def draw_coefficients(rng, model: str, split=(256, 256)):
    """Draw the four coefficient sets (prefill/decode x memory/compute).

    Each coefficient is a roofline-style magnitude times an independent
    jitter exp(0.2 N(0,1)).  Memory-bound segments carry the full weight-load
    cost in beta and a small per-token compute slope; compute-bound segments the
    reverse.  All values are positive.
    """
    wbytes, flop_tok, kv_tok, attn = _COST_SCALES[model]
    coef = np.empty((4, 5), dtype=np.float64)
    for seg in range(4):
        regime = seg & 1
        j = np.exp(0.2 * rng.standard_normal(5))
        if regime == 0:
            base = (wbytes / _BW, 0.05 * flop_tok / _PK, kv_tok / _BW, attn / _PK, 1e-8)
        else:
            base = (0.3 * wbytes / _BW, flop_tok / _PK, kv_tok / _BW, attn / _PK, 1e-8)
        coef[seg] = np.asarray(base) * j
    return coef, np.asarray(split, dtype=np.int64)


def random_batches(rng, n_batch, size_lo, size_hi, prefill_prob, p_law, c_law_decode,
                   n_tenants=16, tenant_s=None, sizes=None):
    """Generic batch generator: per-request Bernoulli phase.

    ``p_law(rng, n)`` draws prefill new-token counts, ``c_law_decode(rng, n)``
    decode contexts.  Prefill requests have c = 0, decode requests p = 1.
    """
    if sizes is None:
        sizes = rng.integers(size_lo, size_hi + 1, size=n_batch, dtype=np.int64)
    off = _offsets_from_sizes(sizes)
    n = int(off[-1])
    phase = (rng.random(n) < prefill_prob).astype(np.int32)
    n_pre = int(phase.sum())
    p = np.ones(n, dtype=np.int32)
    c = np.zeros(n, dtype=np.int32)
    pre = phase == 1
    p[pre] = p_law(rng, n_pre)
    c[~pre] = c_law_decode(rng, n - n_pre)
    if tenant_s is None:
        tenant = rng.integers(0, n_tenants, size=n, dtype=np.int32)
    else:
        tenant = zipf_tenants(rng, n, n_tenants, tenant_s)
    return p, c, phase, tenant, off


def _config0(rng, scale):
    nb = max(1, int(round(20_000 * scale)))
    p, c, ph, t, off = random_batches(
        rng, nb, 1, 64, 0.2,
        lambda r, n: _lognormal_int(r, n, 6.0, 1.0, 1, 8192),
        lambda r, n: r.integers(1, 8193, size=n, dtype=np.int32),
        n_tenants=16)
    return "llama3.1-8b", p, c, ph, t, off, 16


def _config1(rng, scale):
    nb = max(1, int(round(1_000_000 * scale)))
    sizes = rng.integers(16, 257, size=nb, dtype=np.int64)
    off = _offsets_from_sizes(sizes)
    n = int(off[-1])
    k = rng.integers(0, 5, size=nb, dtype=np.int64)          # chunked prefills per batch
    # choose k distinct positions inside each batch, uniformly
    pos = np.empty((nb, 4), dtype=np.int64)
    for j in range(4):
        pos[:, j] = rng.integers(0, sizes)
    while True:
        dup = np.zeros(nb, dtype=bool)
        for a in range(4):
            for b in range(a):
                dup |= (pos[:, a] == pos[:, b]) & (a < k)
        if not dup.any():
            break
        idx = np.nonzero(dup)[0]
        for j in range(4):
            pos[idx, j] = rng.integers(0, sizes[idx])
    phase = np.zeros(n, dtype=np.int32)
    for j in range(4):
        sel = k > j
        phase[off[:-1][sel] + pos[sel, j]] = 1
    pre = phase == 1
    n_pre = int(pre.sum())
    p = np.ones(n, dtype=np.int32)
    c = np.empty(n, dtype=np.int32)
    p[pre] = 512
    c[pre] = rng.integers(0, 32257, size=n_pre, dtype=np.int32)
    c[~pre] = _lognormal_int(rng, n - n_pre, 7.5, 1.2, 1, 32768)
    tenant = zipf_tenants(rng, n, 256, 1.1)
    return "qwen2.5-14b", p, c, phase, tenant, off, 256


def _config2(rng, scale):
    nb = max(1, int(round(2_000_000 * scale)))
    p, c, ph, t, off = random_batches(
        rng, nb, 1, 256, 0.2,
        lambda r, n: _lognormal_int(r, n, 6.0, 1.0, 1, 8192),
        lambda r, n: r.integers(1, 16385, size=n, dtype=np.int32),
        n_tenants=1)
    return "llama3.1-8b", p, c, ph, t, off, 1


def _config4(rng, scale):
    nb = max(1, int(round(10_000_000 * scale)))
    u = 1.0 - rng.random(nb)
    sizes = np.clip(np.floor(u ** (-1.0 / 1.5)), 1, 4096).astype(np.int64)
    p, c, ph, t, off = random_batches(
        rng, nb, 0, 0, 0.1,
        lambda r, n: _log_uniform_int(r, n, 16384),
        lambda r, n: _log_uniform_int(r, n, 131072),
        n_tenants=65536, tenant_s=1.2, sizes=sizes)
    return "llama3.1-8b", p, c, ph, t, off, 65536


_GEN = {0: _config0, 1: _config1, 2: _config2, 4: _config4}


def config(k: int, scale: float = 1.0) -> Workload:
    """Workload ``k`` (0, 1, 2 or 4) with ``scale`` times the number of batches.

    0: Llama3.1-8B tp1, 20,000 batches of U{1..64}, 20 % prefill, 16 tenants.
    1: Qwen2.5-14B tp2, 1e6 continuous-batching batches of U{16..256} with 0-4
       chunked prefills (512 tokens), Zipf(1.1) over 256 tenants.
    2: Llama3.1-8B tp1 fit workload, 2e6 batches of U{1..256}; carries the
       ground-truth coefficients in ``coef`` and lognormal(0, 0.03) noise.
    4: Llama3.1-8B tp1 skew stress, 1e7 Pareto(1.5) batch sizes <= 4096,
       log-uniform contexts, Zipf(1.2) over 65,536 tenants.
    """
    seed = SEED_BASE + k
    rng = np.random.default_rng(seed)
    model, p, c, ph, t, off, nt = _GEN[k](rng, scale)
    coef, split = draw_coefficients(rng, model)
    noise = None
    if k == 2:
        noise = np.exp(0.03 * rng.standard_normal(off.shape[0] - 1))
    return Workload(name=f"config{k}", arch=np.asarray(ARCHS[model], dtype=np.int32), p=p, c=c,
                    phase=ph, tenant=t, offsets=off, n_tenants=nt, coef=coef, split=split,
                    noise=noise, seed=seed)


def step_config(n_req: int = 2048, n_prefill: int = 4) -> Workload:
    """One serving step: a single Qwen2.5-14B tp2 continuous batch of ``n_req``
    requests (the paper's 128-2048 concurrent requests), drawn as in workload 1:
    ``n_prefill`` chunked prefills of 512 new tokens with prior context
    U{0..32256} at random positions, decodes with lognormal(7.5, 1.2) contexts in
    [1, 32768], Zipf(1.1) tenants over 256.
    """
    seed = SEED_BASE + 5
    rng = np.random.default_rng(seed)
    n = int(n_req)
    k = min(int(n_prefill), n)
    phase = np.zeros(n, dtype=np.int32)
    phase[rng.choice(n, size=k, replace=False)] = 1
    pre = phase == 1
    p = np.ones(n, dtype=np.int32)
    c = np.empty(n, dtype=np.int32)
    p[pre] = 512
    c[pre] = rng.integers(0, 32257, size=k, dtype=np.int32)
    c[~pre] = _lognormal_int(rng, n - k, 7.5, 1.2, 1, 32768)
    tenant = zipf_tenants(rng, n, 256, 1.1)
    off = np.array([0, n], dtype=np.int64)
    coef, split = draw_coefficients(rng, "qwen2.5-14b")
    return Workload(name="step", arch=np.asarray(ARCHS["qwen2.5-14b"], dtype=np.int32), p=p, c=c, phase=phase,
                    tenant=tenant, offsets=off, n_tenants=256, coef=coef, split=split, seed=seed)


def whatif_config(scale: float = 1.0, n_pending: int | None = None) -> WhatIf:
    """Workload 3: Qwen2.5-32B tp4 what-if planning.

    1024 candidate batches of U{32..256} requests and 4096 pending requests, each
    request a prefill with probability 0.3; new tokens and contexts follow
    lognormal(8, 1.3) clipped to [1, 131072].
    """
    seed = SEED_BASE + 3
    rng = np.random.default_rng(seed)
    nb = max(1, int(round(1024 * scale)))
    law = lambda r, n: _lognormal_int(r, n, 8.0, 1.3, 1, 131072)  # noqa: E731
    p, c, ph, t, off = random_batches(rng, nb, 32, 256, 0.3, law, law, n_tenants=1)
    npend = n_pending if n_pending is not None else max(1, int(round(4096 * scale)))
    ph_new = (rng.random(npend) < 0.3).astype(np.int32)
    p_new = np.ones(npend, dtype=np.int32)
    c_new = np.zeros(npend, dtype=np.int32)
    pre = ph_new == 1
    p_new[pre] = law(rng, int(pre.sum()))
    c_new[~pre] = law(rng, int((~pre).sum()))
    coef, split = draw_coefficients(rng, "qwen2.5-32b")
    arch = np.asarray(ARCHS["qwen2.5-32b"], dtype=np.int32)
    cand = Workload(name="config3-candidates", arch=arch, p=p, c=c, phase=ph, tenant=t, offsets=off,
                    n_tenants=1, coef=coef, split=split, seed=seed)
    return WhatIf(name="config3", arch=arch, cand=cand, p_new=p_new, c_new=c_new, phase_new=ph_new,
                  coef=coef, split=split, seed=seed)
