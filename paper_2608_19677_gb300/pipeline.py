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

With ``overlap=True`` the planner runs on its own stream and library context:
the plans for interval t+1 depend only on interval t's keys, so they are built
while interval t is routed and replayed and interval t+1 is hashed.  The
planner is latency-bound on a few SMs; the other stages stream over all of
them.  Plans and keys are double-buffered and ordered by CUDA events.
"""
from __future__ import annotations

from typing import Callable, List, Optional, Sequence, Tuple

from . import (Context, Plan, Replay, build_plans, hash_prefixes, plan_params, route_batch,
               shadow_replay)

VARIANT_OF = {"CR": "LPT", "CR_NOLPT": "RANDOM", "CR_NOREPL": "NOREPL"}


class Pipeline:
    def __init__(self, ctx: Context, R: int, W: int, caps: Sequence[int],
                 replicas: Sequence[Tuple[str, int]], qcap: Callable[[int], Tuple[int, int]],
                 batch_B: int = 1024, salt: int = 0, max_n: int = 0, overlap: bool = False):
        import torch
        self.ctx, self.R, self.W, self.caps = ctx, R, W, list(caps)
        self.replicas = list(replicas)
        self.qcap, self.B, self.salt = qcap, batch_B, salt
        self.policies = [p for p, _ in self.replicas]
        self.seeds = [s for _, s in self.replicas]
        dev = torch.device("cuda", ctx.device)
        self.dev = dev
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
        self.overlap = overlap and bool(self.plan_keys)
        if self.overlap:
            self.pstream = torch.cuda.Stream(dev)
            self.pctx = Context(ctx.device, self.pstream)
        else:
            self.pstream, self.pctx = ctx._stream_obj, ctx
        self.plans = [[Plan(self.pctx) for _ in self.plan_keys] for _ in range(2)]
        self.replay = Replay(ctx, len(self.replicas), R, self.caps)
        self.ctr = torch.zeros((len(self.replicas), len(self.caps), R, 5), dtype=torch.int64, device=dev)
        self.load = torch.zeros((len(self.replicas), R), dtype=torch.int64, device=dev)
        self._dest = None
        self._keys = [None, None]
        self._flip = 0
        self.prev_keys = None
        self._ready = [None, None]   # event: plans buffer b is built
        self._pbuf = 0               # plans buffer used by the next interval
        self._next_built = False     # the next interval's plans are already enqueued
        self.plan_marks = []         # (start, end) events of every plan build, when marked
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
        self._next_built = False
        self.plan_marks = []

    def _build(self, buf: int, keys, epoch: int, after, mark: bool):
        """Enqueue the plans of one interval into plans buffer ``buf`` from ``keys``."""
        import torch
        if self.overlap:
            self.pstream.wait_event(after)
        st = self.pstream
        ev0 = torch.cuda.Event(enable_timing=True) if mark else None
        if mark:
            ev0.record(st)
        num, den = self.qcap(int(keys.shape[0]))
        params = [plan_params(self.R, self.W, num, den, v, seed=s, epoch=epoch) for v, s in self.plan_keys]
        build_plans(self.pctx, keys, params, self.plans[buf])
        ready = torch.cuda.Event(enable_timing=mark)
        ready.record(st)
        self._ready[buf] = ready
        if mark:
            self.plan_marks.append((ev0, ready))

    def interval(self, t: int, tokens, off, plen, slen, g0: int, marks=None, plan_next: bool = True):
        """Run one control interval on device tensors; returns the interval's keys.

        ``marks``: optional list of 5 torch.cuda.Event recorded on the main
        stream at the stage boundaries (start, hashed, plans ready, routed,
        replayed); plan builds are timed separately in ``plan_marks``.
        ``plan_next``: with overlap, also enqueue the next interval's plans.
        """
        import torch
        n = int(off.shape[0])
        stream = self.ctx._stream_obj
        if marks is not None:
            marks[0].record(stream)
        self._alloc(n)
        keys = self._keys[self._flip][:n]
        self._flip ^= 1
        hash_prefixes(self.ctx, tokens, off, plen, self.salt, out=keys)
        hashed = torch.cuda.Event()
        hashed.record(stream)
        if marks is not None:
            marks[1].record(stream)
        cur = self._pbuf
        if self.plan_keys:
            if not self._next_built:
                # nothing planned ahead: plan this interval from the previous keys (or its own)
                pk = keys if self.prev_keys is None else self.prev_keys
                self._build(cur, pk, t, hashed, marks is not None)
            if self.overlap and plan_next:
                # the next interval plans from this interval's keys: start now
                self._build(cur ^ 1, keys, t + 1, hashed, marks is not None)
                self._next_built = True
            else:
                self._next_built = False
            if self.overlap:
                stream.wait_event(self._ready[cur])
        if marks is not None:
            marks[2].record(stream)
        self.load.zero_()
        dest = self._dest[:, :n] if n == self._dest.shape[1] else self._dest.view(-1)[:len(self.replicas) * n].view(
            len(self.replicas), n)
        plans = [self.plans[cur][i] if i is not None else None for i in self.rep_plan]
        route_batch(self.ctx, plans, self.policies, self.seeds, self.R, keys, g0, self.B, self.load, dest)
        if marks is not None:
            marks[3].record(stream)
        shadow_replay(self.ctx, self.replay, keys, plen, slen, dest, self.ctr)
        if marks is not None:
            marks[4].record(stream)
        self.prev_keys = keys
        self.last_dest = dest
        self.last_plans = [self.plans[cur][i] for i in range(len(self.plan_keys))]
        if self.overlap and self._next_built:
            self._pbuf = cur ^ 1
        return keys

    def sync(self):
        self.ctx.sync()
        if self.overlap:
            self.pctx.sync()
