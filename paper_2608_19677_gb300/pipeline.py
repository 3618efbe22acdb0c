"""Per-interval driver of the hot path on one GPU (all work in the library's kernels).

One control interval t:
  1. cr_hash_prefixes: routing key of every request;
  2. cr_build_plans: plans from the PREVIOUS interval's keys (the first
     interval plans from its own keys), q_cap from the planning interval's
     request count, one plan per variant in use (LPT for CacheRoute, RANDOM
     seeded per replica for CacheRoute without LPT, NOREPL for single-copy
     CacheRoute), epoch = t;
  3. cr_route_batch: every (policy, seed) replica, loads starting at zero;
  4. cr_shadow_replay: LRU simulators whose state and counters persist over
     intervals.
Keys of interval t stay on the device as the planning input of t+1.
"""
from __future__ import annotations

from typing import Callable, Dict, List, Optional, Sequence, Tuple

from . import (Context, Plan, Replay, build_plans, hash_prefixes, plan_params, route_batch,
               shadow_replay)

VARIANT_OF = {"CR": "LPT", "CR_NOLPT": "RANDOM", "CR_NOREPL": "NOREPL"}


class Pipeline:
    def __init__(self, ctx: Context, R: int, W: int, caps: Sequence[int],
                 replicas: Sequence[Tuple[str, int]], qcap: Callable[[int], Tuple[int, int]],
                 batch_B: int = 1024, salt: int = 0, max_n: int = 0):
        import torch
        self.ctx, self.R, self.W, self.caps = ctx, R, W, list(caps)
        self.replicas = list(replicas)
        self.qcap, self.B, self.salt = qcap, batch_B, salt
        self.policies = [p for p, _ in self.replicas]
        self.seeds = [s for _, s in self.replicas]
        dev = torch.device("cuda", ctx.device)
        # one plan object per distinct (variant, seed) in use
        self.plan_keys: List[Tuple[str, int]] = []
        self.rep_plan: List[Optional[int]] = []
        for p, s in self.replicas:
            v = VARIANT_OF.get(p)
            if v is None:
                self.rep_plan.append(None)
                continue
            k = (v, s if v == "RANDOM" else 0)
            if k not in self.plan_keys:
                self.plan_keys.append(k)
            self.rep_plan.append(self.plan_keys.index(k))
        self.plans = [Plan(ctx) for _ in self.plan_keys]
        self.replay = Replay(ctx, len(self.replicas), R, self.caps)
        self.ctr = torch.zeros((len(self.replicas), len(self.caps), R, 5), dtype=torch.int64, device=dev)
        self.load = torch.zeros((len(self.replicas), R), dtype=torch.int64, device=dev)
        self.dev = dev
        self.prev_keys = None
        self._dest = None
        self._keys = [None, None]
        self._flip = 0
        if max_n:
            self._alloc(max_n)

    def _alloc(self, n: int):
        import torch
        if self._dest is None or self._dest.shape[1] < n:
            self._dest = torch.empty((len(self.replicas), n), dtype=torch.int16, device=self.dev)
            self._keys = [torch.empty(n, dtype=torch.int64, device=self.dev) for _ in range(2)]

    def reset(self):
        self.replay.reset()
        self.ctr.zero_()
        self.prev_keys = None

    def interval(self, t: int, tokens, off, plen, slen, g0: int, marks=None):
        """Run one control interval on device tensors; returns the interval's keys.

        ``marks``: optional list of 5 torch.cuda.Event recorded on the context's
        stream at the stage boundaries (start, hashed, planned, routed, replayed).
        """
        n = int(off.shape[0])
        stream = self.ctx._stream_obj
        if marks is not None:
            marks[0].record(stream)
        self._alloc(n)
        keys = self._keys[self._flip][:n]
        self._flip ^= 1
        hash_prefixes(self.ctx, tokens, off, plen, self.salt, out=keys)
        if marks is not None:
            marks[1].record(stream)
        pk = keys if self.prev_keys is None else self.prev_keys
        if self.plans:
            num, den = self.qcap(int(pk.shape[0]))
            params = [plan_params(self.R, self.W, num, den, v, seed=s, epoch=t) for v, s in self.plan_keys]
            build_plans(self.ctx, pk, params, self.plans)
        if marks is not None:
            marks[2].record(stream)
        self.load.zero_()
        dest = self._dest[:, :n] if n == self._dest.shape[1] else self._dest.view(-1)[:len(self.replicas) * n].view(
            len(self.replicas), n)
        plans = [self.plans[i] if i is not None else None for i in self.rep_plan]
        route_batch(self.ctx, plans, self.policies, self.seeds, self.R, keys, g0, self.B, self.load, dest)
        if marks is not None:
            marks[3].record(stream)
        shadow_replay(self.ctx, self.replay, keys, plen, slen, dest, self.ctr)
        if marks is not None:
            marks[4].record(stream)
        self.prev_keys = keys
        self.last_dest = dest
        return keys
