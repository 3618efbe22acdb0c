"""Seeded synthetic request traces for the planned prefix-affinity router.

This module produces INPUTS only.  It holds none of the routing method's
arithmetic (no prefix hash, no histogram, no plan, no routing rule, no cache
model): it decides which business key each request carries, how long that
key's reusable prefix is, what the prefix tokens are, and how requests are
spread over control intervals.  Both the CPU oracle and the CUDA path consume
exactly the arrays produced here.

Workload shapes follow the paper's description of its traffic (section 2.1 and
the workload table in the supplement: skewed per-key rates, a stable per-key
context that recurs, Poisson or bursty arrivals) at the sizes of the five
synthetic configurations listed in ``CONFIGS``, plus a drift configuration
for the replanning study (sec. 5 "Rate drift and remapping", supplement
"Replanning Under Drift": the 70B-shaped key rates evolve for six intervals by
a lognormal random walk with sigma = 0.3 per step), and a 70B variant whose
arrivals are a Gamma renewal process with inter-arrival CV 1.9 (sec. 5
"Arrival burstiness").  The paper's de-identified
telemetry is not available; these seeded traces stand in for it.

Token values come from a counter-based integer map (``token_values``) over
(stream id, position), evaluated with int64 arithmetic whose products stay
below 2**62, so numpy on the host and torch on a GPU produce the same bytes.
A key's prefix tokens depend only on (trace seed, key id, position); a
request's suffix tokens depend on its global request index.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

VOCAB = 128256
M31 = (1 << 31) - 1

# Policy names (the numeric ids are fixed by the library's public header).
POLICY_IDS = {"CR": 0, "CR_NOLPT": 1, "CR_NOREPL": 2, "P2C": 3, "RR": 4, "HASH": 5, "CHWBL": 6}
SIX_POLICIES = ["CR", "CR_NOLPT", "CR_NOREPL", "P2C", "RR", "HASH"]


def token_values(stream, pos, seed: int = 0, vocab: int = VOCAB, xp=np):
    """Token id for (stream, position): int64 map mod 2**31-1, then mod vocab.

    ``xp`` is numpy or torch; ``stream`` and ``pos`` are int64 arrays/tensors
    of equal shape.  Every product stays below 2**62, so the result is the same
    on any backend.
    """
    x = (stream * 1000003 + pos * 7919 + (seed * 104729 + 12345)) % M31
    x = (x * 48271 + 11) % M31
    x = x ^ (x >> 13)
    x = (x * 69621 + 7) % M31
    x = x ^ (x >> 11)
    x = (x * 48271) % M31
    return x % vocab


@dataclasses.dataclass
class TraceConfig:
    name: str
    R: int                      # destinations
    n_keys: int                 # business keys in the Zipf body
    zipf_s: float
    n_requests: int
    n_intervals: int
    interval_s: float
    plen: Tuple                 # ("fixed", P) | ("lognormal", median, sigma, max) | ("uniform", lo, hi)
    W: int                      # warm slots per destination (C = R*W)
    caps: List[int]             # LRU capacities replayed together
    policies: List[str]
    seeds: List[int]
    suffix: int = 64
    vocab: int = VOCAB
    trace_seed: int = 0
    qcap_mode: str = "mean"     # "mean": q_cap = 1.25 * N/R ; "head": q_cap = N/208 (whale study)
    hot_cap: Optional[float] = None      # water-fill: no key above this share
    whales: Optional[Sequence[int]] = None  # multipliers of injected whale keys
    whale_share: float = 0.25
    burst: Optional[Tuple[float, float, float]] = None  # (factor, burst_len_s, period_s)
    vnodes: int = 64            # ring points per destination of bounded-load (CHWBL) replicas
    drift: Optional[float] = None  # sigma of a per-interval lognormal random walk of every key's rate
    token_caps: Optional[List[int]] = None  # LRU capacities in prefix tokens for the byte-aware replay
    lru_tokens: bool = False    # replay capacities (caps) count prefix tokens instead of prefixes
    arrival_cv: Optional[float] = None  # Gamma renewal arrivals with this inter-arrival CV (else Poisson)

    @property
    def replicas(self) -> List[Tuple[str, int]]:
        return [(p, s) for p in self.policies for s in self.seeds]

    @property
    def total_keys(self) -> int:
        return self.n_keys + (len(self.whales) if self.whales else 0)

    def token_lru(self) -> "TraceConfig":
        """The same workload replayed with token-weighted LRU capacities: ``token_caps``, or
        each prefix-count capacity times the typical prefix length."""
        if self.lru_tokens:
            return self
        if self.token_caps:
            caps = list(self.token_caps)
        else:
            kind = self.plen[0]
            typical = self.plen[1] if kind in ("fixed", "lognormal") else (self.plen[1] + self.plen[2]) // 2
            caps = [c * typical for c in self.caps]
        return dataclasses.replace(self, caps=caps, lru_tokens=True, name=f"{self.name} [token LRU]")

    def scaled(self, n_requests: int, n_intervals: Optional[int] = None, name: Optional[str] = None):
        """Same shape, fewer requests (for sampled or quick runs)."""
        ni = n_intervals if n_intervals is not None else self.n_intervals
        return dataclasses.replace(self, n_requests=n_requests, n_intervals=ni,
                                   name=name or f"{self.name}-n{n_requests}")


CONFIGS: Dict[str, TraceConfig] = {
    "tiny": TraceConfig(
        name="tiny", R=4, n_keys=200, zipf_s=1.1, n_requests=20_000, n_intervals=1,
        interval_s=10.0, plen=("fixed", 512), W=16, caps=[16], policies=["CR", "P2C"],
        seeds=[0]),
    "70b": TraceConfig(
        name="70b", R=30, n_keys=20_000, zipf_s=1.0, n_requests=2_000_000, n_intervals=12,
        interval_s=10.0, plen=("lognormal", 2048, 0.5, 16384), W=12, caps=[12],
        policies=["CR", "P2C", "RR", "HASH"], seeds=[0, 1, 2, 3, 4], hot_cap=1.0 / 30, token_caps=[24576]),
    "8b": TraceConfig(
        name="8b", R=16, n_keys=5_000, zipf_s=1.1, n_requests=4_000_000, n_intervals=800,
        interval_s=10.0, plen=("uniform", 1024, 4096), W=64, caps=[64],
        policies=["CR", "CR_NOLPT", "HASH", "P2C"], seeds=[0, 1, 2], qcap_mode="head",
        whales=[3, 4, 5, 6, 7, 8, 9, 10], whale_share=0.25),
    "burst": TraceConfig(
        name="burst", R=64, n_keys=100_000, zipf_s=0.9, n_requests=16_000_000, n_intervals=120,
        interval_s=5.0, plen=("lognormal", 4096, 0.5, 32768), W=128, caps=[128],
        policies=SIX_POLICIES, seeds=[0, 1, 2, 3, 4], burst=(5.0, 2.0, 30.0)),
    "drift": TraceConfig(
        name="drift", R=30, n_keys=20_000, zipf_s=1.0, n_requests=1_000_000, n_intervals=6,
        interval_s=10.0, plen=("lognormal", 2048, 0.5, 16384), W=12, caps=[12],
        policies=["CR", "P2C"], seeds=[0, 1, 2, 3, 4], hot_cap=1.0 / 30, drift=0.3),
    "70b-gamma": TraceConfig(
        name="70b-gamma", R=30, n_keys=20_000, zipf_s=1.0, n_requests=2_000_000, n_intervals=12,
        interval_s=10.0, plen=("lognormal", 2048, 0.5, 16384), W=12, caps=[12],
        policies=["CR", "P2C", "RR", "HASH"], seeds=[0, 1, 2, 3, 4], hot_cap=1.0 / 30, token_caps=[24576],
        arrival_cv=1.9),
    "large": TraceConfig(
        name="large", R=1024, n_keys=1_000_000, zipf_s=0.8, n_requests=64_000_000,
        n_intervals=60, interval_s=10.0, plen=("lognormal", 2048, 0.5, 32768), W=256,
        caps=[64, 256, 1024], policies=SIX_POLICIES, seeds=list(range(8))),
}


def _rng(seed: int, tag: int, sub: int = 0) -> np.random.Generator:
    """numpy Philox stream keyed by (trace seed, purpose tag, sub-stream)."""
    mask = (1 << 64) - 1
    return np.random.Generator(np.random.Philox(key=[seed & mask, ((tag << 32) ^ sub) & mask]))


def _water_fill(p: np.ndarray, cap: float) -> np.ndarray:
    """Clip shares at ``cap`` and spread the excess over the unclipped keys."""
    p = p.astype(np.float64).copy()
    for _ in range(100):
        over = p > cap
        if not over.any():
            break
        excess = float((p[over] - cap).sum())
        p[over] = cap
        free = ~over & (p < cap)
        p[free] += excess * p[free] / p[free].sum()
    return p / p.sum()


@dataclasses.dataclass
class Interval:
    t: int
    g0: int                 # global index of the first request
    key_id: np.ndarray      # int64 [N]  business key of each request (arrival order)
    plen: np.ndarray        # uint32 [N] prefix tokens
    slen: np.ndarray        # uint32 [N] suffix tokens

    @property
    def n(self) -> int:
        return int(self.key_id.shape[0])


class Trace:
    """Deterministic trace for one configuration; intervals are generated lazily."""

    def __init__(self, cfg: TraceConfig):
        self.cfg = cfg
        self.key_p = self._key_shares()
        self.key_plen = self._key_plens()
        self.counts = self._interval_counts()
        self.g0 = np.concatenate([[0], np.cumsum(self.counts)[:-1]]).astype(np.int64)
        self._cdf = np.cumsum(self.key_p)
        self._cdf[-1] = 1.0
        self._drift_cdf = {}

    # -- key popularity -------------------------------------------------
    def _key_shares(self) -> np.ndarray:
        c = self.cfg
        ranks = np.arange(1, c.n_keys + 1, dtype=np.float64)
        p = ranks ** (-c.zipf_s)
        p /= p.sum()
        if c.hot_cap is not None:
            p = _water_fill(p, c.hot_cap * 0.8)
        if c.whales:
            m = np.asarray(c.whales, dtype=np.float64)
            pw = c.whale_share * m / m.sum()
            p = np.concatenate([p * (1.0 - c.whale_share), pw])
        return p / p.sum()

    def _key_plens(self) -> np.ndarray:
        c = self.cfg
        rng = _rng(c.trace_seed, 0x504C454E)  # "PLEN"
        nk = self.cfg.total_keys
        kind = c.plen[0]
        if kind == "fixed":
            return np.full(nk, c.plen[1], dtype=np.uint32)
        if kind == "uniform":
            return rng.integers(c.plen[1], c.plen[2] + 1, size=nk).astype(np.uint32)
        if kind == "lognormal":
            med, sigma, mx = c.plen[1], c.plen[2], c.plen[3]
            v = np.rint(med * np.exp(sigma * rng.standard_normal(nk)))
            return np.clip(v, 16, mx).astype(np.uint32)
        raise ValueError(kind)

    # -- arrivals ---------------------------------------------------------
    def _interval_counts(self) -> np.ndarray:
        c = self.cfg
        rng = _rng(c.trace_seed, 0x41525256)  # "ARRV"
        secs = int(round(c.n_intervals * c.interval_s))
        if c.arrival_cv:
            t = self.arrival_times()
            idx = np.minimum((t // c.interval_s).astype(np.int64), c.n_intervals - 1)
            return np.bincount(idx, minlength=c.n_intervals).astype(np.int64)
        if c.burst is None:
            w = np.ones(c.n_intervals)
            return rng.multinomial(c.n_requests, w / w.sum()).astype(np.int64)
        factor, blen, period = c.burst
        t = np.arange(secs, dtype=np.float64)
        rate = np.where((t % period) < blen, factor, 1.0)
        per_sec = rng.multinomial(c.n_requests, rate / rate.sum())
        per_int = int(round(c.interval_s))
        return per_sec.reshape(c.n_intervals, per_int).sum(axis=1).astype(np.int64)

    # -- rate drift ---------------------------------------------------------
    def shares(self, t: int) -> np.ndarray:
        """Key shares of interval t.  With drift sigma, every key's log-rate takes an
        independent N(0, sigma^2) step per interval from the primary shares (interval 0),
        and the shares are renormalised (lognormal random walk of the rates)."""
        c = self.cfg
        if not c.drift or t == 0:
            return self.key_p
        walk = np.zeros(c.total_keys)
        for s in range(1, t + 1):
            walk += c.drift * _rng(c.trace_seed, 0x44524654, s).standard_normal(c.total_keys)  # "DRFT"
        p = self.key_p * np.exp(walk)
        return p / p.sum()

    def _cdf_at(self, t: int) -> np.ndarray:
        if not self.cfg.drift or t == 0:
            return self._cdf
        if t not in self._drift_cdf:
            cdf = np.cumsum(self.shares(t))
            cdf[-1] = 1.0
            self._drift_cdf[t] = cdf
        return self._drift_cdf[t]

    def arrival_times(self) -> np.ndarray:
        """Gamma renewal arrivals (configurations with ``arrival_cv``): n gaps of shape
        1/CV^2 (so the gaps' coefficient of variation is arrival_cv), rescaled so the n
        arrivals span the trace; seconds from the trace start."""
        c = self.cfg
        rng = _rng(c.trace_seed, 0x47414D41)  # "GAMA"
        gaps = rng.gamma(1.0 / c.arrival_cv ** 2, 1.0, size=c.n_requests)
        t = np.cumsum(gaps)
        t *= (c.n_intervals * c.interval_s) / (t[-1] * (1.0 + 1e-12))
        return t

    def interval(self, t: int) -> Interval:
        c = self.cfg
        n = int(self.counts[t])
        rng = _rng(c.trace_seed, 0x4B455953, t)  # "KEYS"
        u = rng.random(n)
        kid = np.searchsorted(self._cdf_at(t), u, side="right").astype(np.int64)
        np.minimum(kid, c.total_keys - 1, out=kid)
        plen = self.key_plen[kid]
        slen = np.full(n, c.suffix, dtype=np.uint32)
        return Interval(t=t, g0=int(self.g0[t]), key_id=kid, plen=plen, slen=slen)

    # -- planning inputs that depend only on interval sizes ------------------
    def qcap(self, n_plan: int) -> Tuple[int, int]:
        """q_cap = num/den requests per control interval for a plan built from n_plan requests."""
        c = self.cfg
        if c.qcap_mode == "mean":
            return 5 * max(n_plan, 1), 4 * c.R
        if c.qcap_mode == "head":
            return max(n_plan, 1), 208
        raise ValueError(c.qcap_mode)


# -- token arena ---------------------------------------------------------
def record_layout(iv: Interval, align: int = 4) -> Tuple[np.ndarray, int]:
    """Start offset (in tokens) of each request record and the arena length.

    A record is the request's prefix followed by its suffix, padded to a
    multiple of ``align`` tokens; records are packed in arrival order.
    """
    rec = iv.plen.astype(np.int64) + iv.slen.astype(np.int64)
    rec = (rec + align - 1) // align * align
    off = np.zeros(iv.n, dtype=np.int64)
    if iv.n:
        np.cumsum(rec[:-1], out=off[1:])
    total = int(off[-1] + rec[-1]) if iv.n else 0
    return off.astype(np.uint64), total


def _stream_and_pos(iv: Interval, align: int, n_keys_total: int, xp, device=None):
    """Per-token (stream id, position) for the whole arena of one interval."""
    if xp is np:
        plen = iv.plen.astype(np.int64)
        rec = plen + iv.slen.astype(np.int64)
        rec = (rec + align - 1) // align * align
        req = np.repeat(np.arange(iv.n, dtype=np.int64), rec)
        start = np.zeros(iv.n, dtype=np.int64)
        if iv.n:
            np.cumsum(rec[:-1], out=start[1:])
        j = np.arange(req.shape[0], dtype=np.int64) - start[req]
        in_prefix = j < plen[req]
        stream = np.where(in_prefix, iv.key_id[req],
                          n_keys_total + iv.g0 + req)
        pos = np.where(in_prefix, j, j - plen[req])
        return stream, pos
    import torch
    plen = torch.as_tensor(iv.plen.astype(np.int64), device=device)
    slen = torch.as_tensor(iv.slen.astype(np.int64), device=device)
    kid = torch.as_tensor(iv.key_id, device=device)
    rec = (plen + slen + align - 1) // align * align
    req = torch.repeat_interleave(torch.arange(iv.n, device=device, dtype=torch.int64), rec)
    start = torch.cumsum(rec, 0) - rec
    j = torch.arange(req.shape[0], device=device, dtype=torch.int64) - start[req]
    preq = plen[req]
    in_prefix = j < preq
    stream = torch.where(in_prefix, kid[req], n_keys_total + iv.g0 + req)
    pos = torch.where(in_prefix, j, j - preq)
    return stream, pos


def arena_host(trace: Trace, iv: Interval, align: int = 4):
    """(tokens int32[T], off uint64[N]) on the host.

    Each distinct key's prefix span is evaluated once and copied into every
    record that carries it; suffix and padding tokens are evaluated per record.
    Same bytes as ``arena_device``.
    """
    cfg = trace.cfg
    off, total = record_layout(iv, align)
    out = np.empty(total, dtype=np.int32)
    if iv.n == 0:
        return out, off
    # suffix + padding: every position of a record at or after its prefix
    plen = iv.plen.astype(np.int64)
    rec = plen + iv.slen.astype(np.int64)
    rec = (rec + align - 1) // align * align
    tail = rec - plen
    req = np.repeat(np.arange(iv.n, dtype=np.int64), tail)
    tstart = np.zeros(iv.n, dtype=np.int64)
    np.cumsum(tail[:-1], out=tstart[1:])
    j = np.arange(req.shape[0], dtype=np.int64) - tstart[req]
    tail_tok = token_values(cfg.total_keys + iv.g0 + req, j, cfg.trace_seed, cfg.vocab)
    out[(off.astype(np.int64)[req] + plen[req] + j)] = tail_tok.astype(np.int32)
    # prefixes
    cache = {}
    o = off.astype(np.int64)
    for i in range(iv.n):
        k = int(iv.key_id[i])
        pt = cache.get(k)
        if pt is None:
            pt = prefix_tokens(trace, k)
            cache[k] = pt
        out[o[i]:o[i] + pt.shape[0]] = pt
    return out, off


def arena_device(trace: Trace, iv: Interval, align: int = 4, device="cuda", chunk_req: int = 1 << 16):
    """(tokens int32[T], off uint64-as-int64[N]) built on ``device`` with torch ops.

    Produces the same bytes as ``arena_host``; built in request chunks to bound
    temporary memory.
    """
    import torch
    off, total = record_layout(iv, align)
    out = torch.empty(total, dtype=torch.int32, device=device)
    for a in range(0, iv.n, chunk_req):
        b = min(iv.n, a + chunk_req)
        sub = Interval(t=iv.t, g0=iv.g0 + a, key_id=iv.key_id[a:b], plen=iv.plen[a:b],
                       slen=iv.slen[a:b])
        stream, pos = _stream_and_pos(sub, align, trace.cfg.total_keys, torch, device)
        tok = token_values(stream, pos, trace.cfg.trace_seed, trace.cfg.vocab, xp=torch)
        lo = int(off[a])
        out[lo:lo + tok.shape[0]] = tok.to(torch.int32)
    return out, torch.as_tensor(off.view(np.int64), device=device)


_ctok = None


def _tokens_lib():
    """The C token generator (compiled on first use with the host C compiler)."""
    global _ctok
    if _ctok is None:
        import ctypes
        import os
        import subprocess
        here = os.path.dirname(os.path.abspath(__file__))
        src, lib = os.path.join(here, "_tokens.c"), os.path.join(here, "_tokens.so")
        if not os.path.exists(lib) or os.path.getmtime(lib) < os.path.getmtime(src):
            tmp = lib + f".tmp{os.getpid()}"
            subprocess.check_call(["gcc", "-std=c11", "-O2", "-fPIC", "-shared", "-o", tmp, src])
            os.replace(tmp, lib)
        L = ctypes.CDLL(lib)
        L.tg_prefix_tokens.restype = None
        L.tg_prefix_tokens.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int64,
                                       ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_uint64]
        _ctok = L
    return _ctok


def prefix_spans(trace: Trace, key_ids) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Prefix spans of many keys packed back to back: (tokens int32, off uint64, plen uint32)."""
    ids = np.ascontiguousarray(key_ids, dtype=np.int64)
    pl = np.ascontiguousarray(trace.key_plen[ids], dtype=np.uint32)
    total = int(pl.astype(np.int64).sum())
    tok = np.empty(max(total, 1), dtype=np.int32)
    off = np.empty(max(ids.size, 1), dtype=np.uint64)
    start = np.zeros(ids.size + 1, dtype=np.int64)
    np.cumsum(pl, out=start[1:])
    L = _tokens_lib()

    def fill(ab):  # keys [a, b) into their slice of the arena (the C call releases the GIL)
        a, b = ab
        if b > a:
            L.tg_prefix_tokens(ids.ctypes.data + 8 * a, pl.ctypes.data + 4 * a, b - a, trace.cfg.trace_seed,
                               trace.cfg.vocab, tok.ctypes.data + 4 * int(start[a]), off.ctypes.data + 8 * a,
                               int(start[a]))

    import concurrent.futures as cf
    import os
    nt = max(1, min(os.cpu_count() or 1, 16, ids.size // 256 + 1))
    cuts = [ids.size * i // nt for i in range(nt + 1)]
    with cf.ThreadPoolExecutor(nt) as ex:
        list(ex.map(fill, zip(cuts[:-1], cuts[1:])))
    return tok[:total], off[:ids.size], pl


def prefix_tokens(trace: Trace, key_id: int) -> np.ndarray:
    """The prefix token span of one business key (host)."""
    p = int(trace.key_plen[key_id])
    pos = np.arange(p, dtype=np.int64)
    stream = np.full(p, key_id, dtype=np.int64)
    return token_values(stream, pos, trace.cfg.trace_seed, trace.cfg.vocab).astype(np.int32)


def random_dest(n_rep: int, n: int, R: int, seed: int) -> np.ndarray:
    """Arbitrary destination assignments (uint16 [n_rep, n]) for testing the replay alone."""
    rng = _rng(seed, 0x44455354)
    return rng.integers(0, R, size=(n_rep, n)).astype(np.uint16)
