"""The oracle's multi-interval protocol (TEST INFRASTRUCTURE ONLY).

One control interval t of a trace:
  1. hash every request's prefix span into its routing key;
  2. build the plan from the PREVIOUS interval's keys (interval 0, which has no
     predecessor, plans from its own keys; with ``fresh`` every interval plans
     from its own keys: the fresh plan of the stale-vs-fresh comparison in the
     supplement "Replanning Under Drift"); q_cap = 1.25 x the mean
     destination load of the planning interval (or N/208 for the whale study);
     one plan per variant: LPT for CacheRoute, RANDOM (seeded) for CacheRoute
     without LPT, NOREPL for single-copy CacheRoute; epoch = t;
  3. route the interval for every (policy, seed) replica with loads starting
     at zero, in batches of B;
  4. replay the routed requests through every LRU simulator; simulator state
     and counters persist from interval to interval.
"""
from __future__ import annotations

import time
from typing import Iterable, Optional

import numpy as np

import tracegen as tg
from . import Replay, Ring, build_plan, hash_prefixes, route

VARIANT_OF = {"CR": "LPT", "CR_NOLPT": "RANDOM", "CR_NOREPL": "NOREPL", "CR_SLOTCAP": "SLOTCAP"}
ROUTE_AS = {"CR_SLOTCAP": "CR"}  # routed as CacheRoute on the slot-capped plan


def plans_for_interval(trace: tg.Trace, plan_keys: np.ndarray, t: int):
    cfg = trace.cfg
    num, den = trace.qcap(int(plan_keys.shape[0]))
    built = {}
    per_rep = []
    for pol, seed in cfg.replicas:
        v = VARIANT_OF.get(pol)
        if v is None:
            per_rep.append(None)
            continue
        k = (v, seed if v == "RANDOM" else 0)
        if k not in built:
            built[k] = build_plan(plan_keys, cfg.R, cfg.W, num, den, variant=v,
                                  seed=k[1], epoch=t)
        per_rep.append(built[k])
    return per_rep, built


def rings_for(cfg):
    """Ring of every bounded-load (CHWBL) replica, seeded by the replica's seed; None elsewhere."""
    return [Ring(cfg.R, cfg.vnodes, seed) if pol == "CHWBL" else None for pol, seed in cfg.replicas]


def run_trace(trace: tg.Trace, intervals: Optional[Iterable[int]] = None, align: int = 4,
              B: int = 1024, salt: int = 0, keep: bool = False, time_budget_s: Optional[float] = None,
              fresh: bool = False):
    """Run the protocol; returns a dict with the counters (and per-interval data if keep)."""
    cfg = trace.cfg
    reps = cfg.replicas
    pols = [ROUTE_AS.get(p, p) for p, _ in reps]
    seeds = [s for _, s in reps]
    rp = Replay(len(reps), cfg.R, cfg.caps, tokens=cfg.lru_tokens)
    rings = rings_for(cfg)
    prev = None
    out = {"intervals": [], "keys": [], "plans": [], "dest": [], "load": [], "requests": 0}
    t_start = time.perf_counter()
    for t in (range(cfg.n_intervals) if intervals is None else intervals):
        iv = trace.interval(t)
        tok, off = tg.arena_host(trace, iv, align)
        keys = hash_prefixes(tok, off, iv.plen, salt)
        per_rep, built = plans_for_interval(trace, keys if (prev is None or fresh) else prev, t)
        dest, load = route(per_rep, pols, seeds, cfg.R, keys, iv.g0, B, rings=rings)
        rp.step(keys, iv.plen, iv.slen, dest)
        prev = keys
        out["intervals"].append(t)
        out["requests"] += iv.n
        if keep:
            out["keys"].append(keys)
            out["plans"].append(built)
            out["dest"].append(dest)
            out["load"].append(load)
        if time_budget_s is not None and time.perf_counter() - t_start > time_budget_s:
            break
    out["ctr"] = rp.ctr.copy()
    out["replay"] = rp
    return out
