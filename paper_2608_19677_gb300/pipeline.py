"""Per-interval driver of the hot path on one GPU (all work in the library's kernels).

One control interval t:
  1. cr_hash_prefixes: routing key of every request;
  2. cr_build_plans: plans from the PREVIOUS interval's keys (the first
     interval plans from its own keys; with ``fresh`` every interval plans
     from its own keys, as in the paper's stale-vs-fresh replanning
     comparison), q_cap from the planning interval's
     request count, one plan per variant in use (LPT for CacheRoute, RANDOM
     seeded per replica for CacheRoute without LPT, NOREPL for single-copy
     CacheRoute), epoch = t;
  3. cr_route_batch: every (policy, seed) replica, loads starting at zero
     (bounded-load replicas use a ring built once, seeded by the replica);
  4. cr_shadow_replay: LRU simulators whose state and counters persist over
     intervals (capacities in prefixes, or with ``lru_tokens`` in prefix tokens).

With ``overlap=True`` the planner runs on its own high-priority stream and
library context, ordered by CUDA events: plans(t+1) need only interval t's
keys, so they are built on a few SMs while interval t is routed and replayed
and interval t+1 is hashed on the main stream.  The replay also has a stream
and context of its own: replay(t) needs only interval t's destinations, so it
runs while interval t+1 is hashed and routed.  (The driver can also put
hashing on a stream of its own; that is off because the hash kernel's CTAs
occupy every SM and would delay the single-SM routing CTAs instead of sharing
the machine with them.)  Keys are triple-buffered, plans and destinations
double-buffered; a buffer is reused only after events show its last reader has
finished.  ``inputs_free`` is the event after which the last interval's input
tensors are no longer read.
"""
from __future__ import annotations

from typing import Callable, List, Optional, Sequence, Tuple

from . import (Context, Plan, Replay, ReplayInput, Ring, build_plans, hash_prefixes, plan_params, replay_partition,
               replay_simulate, route_batch, set_resolve_stream, shadow_replay)

VARIANT_OF = {"CR": "LPT", "CR_NOLPT": "RANDOM", "CR_NOREPL": "NOREPL", "CR_SLOTCAP": "SLOTCAP"}
# CacheRoute on a slot-capped plan routes as CacheRoute (same fallback draws as CR, seed for seed)
ROUTE_AS = {"CR_SLOTCAP": "CR"}
NKEYS = 3


class Pipeline:
    def __init__(self, ctx: Context, R: int, W: int, caps: Sequence[int],
                 replicas: Sequence[Tuple[str, int]], qcap: Callable[[int], Tuple[int, int]],
                 batch_B: int = 1024, salt: int = 0, max_n: int = 0, overlap: bool = False,
                 vnodes: int = 64, fresh: bool = False, lru_tokens: bool = False, resolve_stream=None):
        import torch
        self.ctx, self.R, self.W, self.caps = ctx, R, W, list(caps)
        self.replicas = list(replicas)
        self.qcap, self.B, self.salt = qcap, batch_B, salt
        self.fresh = fresh  # plans from each interval's own keys instead of the previous interval's
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
        self.overlap = overlap
        self.mstream = ctx._stream_obj
        if overlap:
            # Hashing stays on the main stream: its CTAs fill every SM, so a
            # hash stream would starve the single-SM routing CTAs rather than
            # share with them.  The planner gets its own high-priority stream.
            lo, hi = torch.cuda.Stream.priority_range() if hasattr(torch.cuda.Stream, "priority_range") else (0, -1)
            self.hstream, self.hctx = self.mstream, ctx
            self.pstream = torch.cuda.Stream(dev, priority=hi)
            self.pctx = Context(ctx.device, self.pstream)
            self.ystream = torch.cuda.Stream(dev)
            self.yctx = Context(ctx.device, self.ystream)
        else:
            self.hstream = self.pstream = self.ystream = self.mstream
            self.hctx = self.pctx = self.yctx = ctx
        # split routing: the load-dependent resolution on a stream of its own (e.g. a small SM
        # partition), so that it overlaps the next interval's hashing on the main stream
        self.xstream = resolve_stream if overlap else None
        self.plans = [[Plan(self.pctx) for _ in self.plan_keys] for _ in range(2)]
        self.replay = Replay(ctx, len(self.replicas), R, self.caps, tokens=lru_tokens)
        # ring of every bounded-load replica, seeded by the replica's seed (built once)
        self.rings = [Ring(ctx, R, vnodes, s) if p == "CHWBL" else None for p, s in self.replicas]
        self.ctr = torch.zeros((len(self.replicas), len(self.caps), R, 5), dtype=torch.int64, device=dev)
        self.load = torch.zeros((len(self.replicas), R), dtype=torch.int64, device=dev)
        self._dests = [None, None]   # destinations, double-buffered when the replay lags
        self._dest_free = [None, None]  # event: the replay that read this buffer has finished
        self._dbuf = 0
        self.inputs_free = None
        self._keys = [None] * NKEYS
        self._released = [[] for _ in range(NKEYS)]  # events after which a keys buffer may be rewritten
        self._kidx = 0
        self.prev_keys = None
        self._prev_kb = None
        self._ready = [None, None]   # event: plans buffer b is built
        self._plan_free = [None, None]  # event: the route that read plans buffer b has finished
        self._routed_prev = None     # event: the last route call's end (split routing)
        self._pbuf = 0               # plans buffer used by the next interval
        self._next_built = False     # the next interval's plans are already enqueued
        self.plan_marks = []         # (start, end) events of every plan build, when marked
        self.hash_marks = []         # (start, end) events of every hash, when marked
        self.route_marks = []        # (start, end) events of every route call, after its waits
        self.replay_marks = []       # (start, end) events of every replay call, after its waits
        if max_n:
            self._alloc(max_n)

    @property
    def contexts(self):
        out = []
        for c in (self.ctx, self.hctx, self.pctx, self.yctx):
            if all(c is not o for o in out):
                out.append(c)
        return out

    def _alloc(self, n: int):
        import torch
        if self._dests[0] is None or self._dests[0].shape[1] < n:
            self.sync()
            nd = 2 if self.overlap else 1
            self._dests = [torch.empty((len(self.replicas), n), dtype=torch.int16, device=self.dev)
                           for _ in range(nd)] + [None] * (2 - nd)
            self._dest_free = [None, None]
            self._keys = [torch.empty(n, dtype=torch.int64, device=self.dev) for _ in range(NKEYS)]
            self._released = [[] for _ in range(NKEYS)]

    def reset(self):
        """Empty the simulators and counters; later work is ordered after everything before."""
        import torch
        self.replay.reset()
        self.ctr.zero_()
        self.prev_keys = None
        self._prev_kb = None
        self._next_built = False
        self.plan_marks = []
        self.hash_marks = []
        self.route_marks = []
        self.replay_marks = []
        if self.overlap:
            start = torch.cuda.Event()
            start.record(self.mstream)
            self.hstream.wait_event(start)
            self.pstream.wait_event(start)
            self.ystream.wait_event(start)

    def _event(self, stream, timing=False):
        import torch
        e = torch.cuda.Event(enable_timing=timing)
        e.record(stream)
        return e

    def _build(self, buf: int, keys, epoch: int, after, mark: bool):
        """Enqueue the plans of one interval into plans buffer ``buf`` from ``keys``."""
        if self.overlap:
            self.pstream.wait_event(after)
            if self._plan_free[buf] is not None:  # the route that last read this buffer
                self.pstream.wait_event(self._plan_free[buf])
        ev0 = self._event(self.pstream, True) if mark else None
        num, den = self.qcap(int(keys.shape[0]))
        params = [plan_params(self.R, self.W, num, den, v, seed=s, epoch=epoch) for v, s in self.plan_keys]
        build_plans(self.pctx, keys, params, self.plans[buf])
        ready = self._event(self.pstream, mark)
        self._ready[buf] = ready
        if mark:
            self.plan_marks.append((ev0, ready))
        return ready

    def interval(self, t: int, tokens, off, plen, slen, g0: int, marks=None, plan_next: bool = True,
                 inputs_ready=None, keys=None):
        """Enqueue one control interval on device tensors; returns the interval's keys.

        ``marks``: optional list of 5 torch.cuda.Event recorded on the main
        stream at the stage boundaries (start, keys ready, plans ready, routed,
        replayed); hash and plan builds are timed in ``hash_marks`` and
        ``plan_marks`` on their own streams.  ``plan_next``: with overlap, also
        enqueue the next interval's plans.  ``inputs_ready``: event after which
        the input tensors may be read (e.g. the end of their copy).  ``keys``:
        the interval's routing keys when they were computed beforehand (the
        token arena is then not read and may be None).
        """
        import torch
        n = int(keys.shape[0]) if keys is not None else int(off.shape[0])
        mark = marks is not None
        if mark:
            marks[0].record(self.mstream)
        self._alloc(n)
        kb = self._kidx
        self._kidx = (self._kidx + 1) % NKEYS
        # ---- hash ---------------------------------------------------------------
        for e in self._released[kb]:
            self.hstream.wait_event(e)
        self._released[kb] = []
        if inputs_ready is not None:
            self.hstream.wait_event(inputs_ready)
        if keys is None:
            keys = self._keys[kb][:n]
            h0 = self._event(self.hstream, True) if mark else None
            hash_prefixes(self.hctx, tokens, off, plen, self.salt, out=keys)
            hashed = self._event(self.hstream, mark)
            if mark:
                self.hash_marks.append((h0, hashed))
        else:
            hashed = self._event(self.hstream)
        # ---- plans ----------------------------------------------------------------
        cur = self._pbuf
        plan_reader = None
        if self.plan_keys and self.fresh:
            # a freshly computed plan: this interval's own keys (replanning study)
            plan_reader = self._build(cur, keys, t, hashed, mark)
            self._next_built = False
        elif self.plan_keys:
            if not self._next_built:
                # nothing planned ahead: plan this interval from the previous keys (or its own)
                if self.prev_keys is None:
                    pk, after = keys, hashed
                else:
                    pk, after = self.prev_keys, self._prev_hashed
                built = self._build(cur, pk, t, after, mark)
                if self.overlap and self.prev_keys is not None:
                    self._released[self._prev_kb].append(built)
            if self.overlap and plan_next:
                # the next interval plans from this interval's keys: start as soon as they exist
                plan_reader = self._build(cur ^ 1, keys, t + 1, hashed, mark)
                self._next_built = True
            else:
                self._next_built = False
        # ---- route and replay ---------------------------------------------------------
        if self.overlap:
            self.mstream.wait_event(hashed)
            if self.plan_keys:
                self.mstream.wait_event(self._ready[cur])
        if mark:
            marks[1].record(self.mstream)
            marks[2].record(self.mstream)
        if self.xstream is not None and self._routed_prev is not None:
            self.mstream.wait_event(self._routed_prev)  # the last resolution wrote the loads
        with torch.cuda.stream(self.mstream):
            self.load.zero_()
        db = self._dbuf
        if self.overlap:
            self._dbuf ^= 1
            if self._dest_free[db] is not None:
                self.mstream.wait_event(self._dest_free[db])
        D = self._dests[db]
        dest = D[:, :n] if n == D.shape[1] else D.view(-1)[:len(self.replicas) * n].view(len(self.replicas), n)
        plans = [self.plans[cur][i] if i is not None else None for i in self.rep_plan]
        r0 = self._event(self.mstream, True) if mark else None
        # the split is a property of the library context, which other pipelines may share:
        # set it for every call (the library synchronises only when it changes)
        set_resolve_stream(self.ctx, self.xstream)
        route_batch(self.ctx, plans, [ROUTE_AS.get(p, p) for p in self.policies], self.seeds, self.R, keys, g0,
                    self.B, self.load, dest, rings=self.rings)
        rstream = self.xstream if self.xstream is not None else self.mstream  # where the route call ends
        if mark:
            marks[3].record(rstream)
            self.route_marks.append((r0, marks[3]))
        if self.overlap:
            routed = self._event(rstream)
            self.ystream.wait_event(routed)
            if self.xstream is not None:
                self._plan_free[cur] = routed
                self._routed_prev = routed
        y0 = self._event(self.ystream, True) if mark else None
        shadow_replay(self.yctx, self.replay, keys, plen, slen, dest, self.ctr)
        replayed = self._event(self.ystream, mark)
        if mark:
            marks[4].record(self.ystream)
            self.replay_marks.append((y0, replayed))
        self.inputs_free = replayed
        # keys buffer kb is free once this interval's replay and the next plans have read it
        if self.overlap:
            self._dest_free[db] = replayed
            self._released[kb].append(replayed)
            if plan_reader is not None:
                self._released[kb].append(plan_reader)
        self.prev_keys = keys
        self._prev_kb = kb
        self._prev_hashed = hashed
        self.last_dest = dest
        self.last_plans = [self.plans[cur][i] for i in range(len(self.plan_keys))]
        if self.overlap and self._next_built:
            self._pbuf = cur ^ 1
        return keys

    def wait_last(self):
        """Make torch's current stream wait for everything enqueued so far on the
        pipeline's streams, so that ``last_dest`` and the counters can be read on it
        whatever stream the caller uses; the host does not block."""
        import torch
        cur = torch.cuda.current_stream(self.dev)
        for st in (self.mstream, self.pstream, self.ystream) + ((self.xstream,) if self.xstream is not None else ()):
            cur.wait_event(self._event(st))

    def quiesce(self):
        """Wait for all enqueued work and forget the events that ordered it, so the next
        interval waits on nothing recorded before (e.g. before capturing a CUDA graph)."""
        self.sync()
        self._released = [[] for _ in range(NKEYS)]
        self._dest_free = [None, None]
        self._ready = [None, None]
        self._plan_free = [None, None]
        self._routed_prev = None
        self._next_built = False
        self.inputs_free = None

    def finish(self):
        """Make the main stream wait for every other stream's enqueued work."""
        if self.overlap:
            self.mstream.wait_event(self._event(self.hstream))
            self.mstream.wait_event(self._event(self.pstream))
            self.mstream.wait_event(self._event(self.ystream))
            if self.xstream is not None:
                self.mstream.wait_event(self._event(self.xstream))

    def close(self):
        """Free the pipeline's plans, replay state and rings, close the contexts it created,
        and detach the caller's context from the resolve stream, in that order (so that a
        stream the pipeline was given, e.g. of an SM partition, can be destroyed afterwards)."""
        self.sync()
        for buf in self.plans:
            for pl in buf:
                pl.close()
        self.replay.close()
        for g in self.rings:
            if g is not None:
                g.close()
        if self.xstream is not None:
            set_resolve_stream(self.ctx, None)
        for c in self.contexts:
            if c is not self.ctx:
                c.close()

    def sync(self):
        if self.xstream is not None:
            self.xstream.synchronize()
        for c in self.contexts:
            c.sync()

    @property
    def launches(self) -> int:
        return sum(c.launches for c in self.contexts)


class TracePipeline:
    """Offline shadow replay of a whole trace whose routing keys are already on the device.

    The plan of interval t depends only on interval t-1's keys, and routing
    starts every interval from zero loads, so plans and routes of different
    intervals are independent; only the replay, whose LRU state carries over,
    must take the intervals in order.  This driver therefore keeps ``depth``
    intervals in flight: plan builds go round-robin to ``plan_streams``
    streams (each with its own library context and scratch), routing to
    ``route_streams`` streams, and the replay of interval t follows its route
    on one replay stream.  Plan and destination buffers are reused every
    ``depth`` intervals, each reuse ordered by the event of its last reader.
    The results equal the per-interval ``Pipeline``'s (same plans, routes and
    counters); only the schedule differs.
    """

    def __init__(self, ctx: Context, R: int, W: int, caps: Sequence[int],
                 replicas: Sequence[Tuple[str, int]], qcap: Callable[[int], Tuple[int, int]],
                 max_n: int, batch_B: int = 1024, depth: int = 8, plan_streams: int = 4,
                 route_streams: int = 4, vnodes: int = 64, fresh: bool = False, lru_tokens: bool = False,
                 replay_first: bool = False, replay_group: int = 1):
        import torch
        self.ctx, self.R, self.W, self.caps = ctx, R, W, list(caps)
        self.replicas = list(replicas)
        self.qcap, self.B, self.fresh = qcap, batch_B, fresh
        self.policies = [ROUTE_AS.get(p, p) for p, _ in self.replicas]
        self.seeds = [s for _, s in self.replicas]
        self.dev = torch.device("cuda", ctx.device)
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
        self.depth = max(1, depth)
        self.mstream = ctx._stream_obj
        # The replay is the one serial chain (interval after interval); with
        # ``replay_first`` its stream has the high priority, so that its kernels take
        # SMs ahead of the plans and routes of later intervals, which have slack.
        lo, hi = torch.cuda.Stream.priority_range() if hasattr(torch.cuda.Stream, "priority_range") else (0, -1)
        self.pstreams = [torch.cuda.Stream(self.dev, priority=lo if replay_first else hi)
                         for _ in range(max(1, plan_streams))]
        self.pctxs = [Context(ctx.device, s) for s in self.pstreams]
        self.rstreams = [torch.cuda.Stream(self.dev, priority=lo) for _ in range(max(1, route_streams))]
        self.rctxs = [Context(ctx.device, s) for s in self.rstreams]
        self.ystream = torch.cuda.Stream(self.dev, priority=hi if replay_first else lo)
        self.yctx = Context(ctx.device, self.ystream)
        self.plans = [[Plan(self.pctxs[0]) for _ in self.plan_keys] for _ in range(self.depth)]
        self.replay = Replay(ctx, len(self.replicas), R, self.caps, tokens=lru_tokens)
        self.rings = [Ring(ctx, R, vnodes, s) if p == "CHWBL" else None for p, s in self.replicas]
        nrep = len(self.replicas)
        self.ctr = torch.zeros((nrep, len(self.caps), R, 5), dtype=torch.int64, device=self.dev)
        self.loads = [torch.zeros((nrep, R), dtype=torch.int64, device=self.dev) for _ in self.rstreams]
        self.max_n = max_n
        self.dests = [torch.empty(nrep * max_n, dtype=torch.int16, device=self.dev) for _ in range(self.depth)]
        # grouped replay: `replay_group` consecutive intervals are staged into one buffer
        # (inputs and destinations, [replica][request of the group]) and replayed by one
        # call, which pays the per-stream setup of the replay once per group
        self.group = max(1, replay_group)
        self.inputs = [ReplayInput(ctx) for _ in range(2)]  # partitioned groups, double-buffered
        self.gbuf = []
        if self.group > 1:
            G = self.group * max_n
            for _ in range(2):
                self.gbuf.append((torch.empty(G, dtype=torch.int64, device=self.dev),
                                  torch.empty(G, dtype=torch.int32, device=self.dev),
                                  torch.empty(G, dtype=torch.int32, device=self.dev),
                                  torch.empty(nrep * G, dtype=torch.int16, device=self.dev)))
        ctx.sync()
        self._reset_events()
        self.plan_marks, self.route_marks, self.replay_marks = [], [], []

    def _reset_events(self):
        self._plan_free = [None] * self.depth   # route that last read plans buffer b
        self._dest_free = [None] * self.depth   # replay that last read destinations buffer b
        self._load_free = [None] * len(self.rstreams)
        self._gfree = [None, None]              # replay that last read group buffer k

    @property
    def contexts(self):
        return [self.ctx] + self.pctxs + self.rctxs + [self.yctx]

    @property
    def launches(self) -> int:
        return sum(c.launches for c in self.contexts)

    def _event(self, stream, timing=False):
        import torch
        e = torch.cuda.Event(enable_timing=timing)
        e.record(stream)
        return e

    def dest_view(self, b: int, n: int):
        return self.dests[b][:len(self.replicas) * n].view(len(self.replicas), n)

    def run(self, keys, plens, slens, g0s, mark: bool = False, on_interval=None, ready=None):
        """Enqueue every interval of the trace (lists of device tensors and first request
        indices) after the work already on the main stream; the main stream then waits for
        all of it.  Counters accumulate in ``ctr`` (call ``reset`` between runs).
        ``ready[t]``, when given, is an event after which interval t's tensors may be read
        (e.g. the end of their host-to-device copy).
        ``on_interval(t, dest, plans)``, when given, is called after interval t is enqueued
        with its destinations view and plans (a test hook: the caller must order its reads
        after the pipeline's streams, e.g. by ``sync``, before the buffer's reuse)."""
        import torch
        T = len(keys)
        start = self._event(self.mstream)
        for s in self.pstreams + self.rstreams + [self.ystream]:
            s.wait_event(start)
        self.plan_marks, self.route_marks, self.replay_marks, self.part_marks = [], [], [], []
        # replay groups: [g0, g1) intervals, their request count, and each interval's column
        sizes = [int(k.shape[0]) for k in keys]
        groups, col = [], [0] * T
        for g0 in range(0, T, self.group):
            g1 = min(T, g0 + self.group)
            c = 0
            for t in range(g0, g1):
                col[t] = c
                c += sizes[t]
            groups.append((g0, g1, c))
        staged = []
        for t in range(T):
            n = int(keys[t].shape[0])
            if n > self.max_n:
                raise ValueError(f"interval {t} has {n} requests, more than max_n={self.max_n}")
            b = t % self.depth
            # ---- plans of interval t (from interval t-1's keys; interval 0 from its own) ----
            plans = None
            if self.plan_keys:
                ps = self.pstreams[t % len(self.pstreams)]
                pc = self.pctxs[t % len(self.pctxs)]
                if self._plan_free[b] is not None:
                    ps.wait_event(self._plan_free[b])
                pt = t if (t == 0 or self.fresh) else t - 1
                pk = keys[pt]
                if ready is not None:
                    ps.wait_event(ready[pt])
                num, den = self.qcap(int(pk.shape[0]))
                params = [plan_params(self.R, self.W, num, den, v, seed=s, epoch=t) for v, s in self.plan_keys]
                p0 = self._event(ps, True) if mark else None
                build_plans(pc, pk, params, self.plans[b])
                built = self._event(ps, mark)
                if mark:
                    self.plan_marks.append((p0, built))
                plans = [self.plans[b][i] if i is not None else None for i in self.rep_plan]
            # ---- route of interval t ---------------------------------------------------
            q = t % len(self.rstreams)
            rs, rc = self.rstreams[q], self.rctxs[q]
            if plans is not None:
                rs.wait_event(built)
            if self._dest_free[b] is not None:
                rs.wait_event(self._dest_free[b])
            if ready is not None:
                rs.wait_event(ready[t])  # the replay follows the route, so it sees the inputs too
            dest = self.dest_view(b, n)
            r0 = self._event(rs, True) if mark else None
            with torch.cuda.stream(rs):
                self.loads[q].zero_()
            route_batch(rc, plans if plans is not None else [None] * len(self.replicas), self.policies,
                        self.seeds, self.R, keys[t], g0s[t], self.B, self.loads[q], dest, rings=self.rings)
            routed = self._event(rs, mark)
            if mark:
                self.route_marks.append((r0, routed))
            self._plan_free[b] = routed
            if on_interval is not None:
                on_interval(t, dest, self.plans[b] if self.plan_keys else [])
            # ---- replay: partition on the route stream, simulation in interval order ---------
            # (the partition of later intervals runs while the simulators work through
            # earlier ones; only the simulation carries state from interval to interval)
            gi = t // self.group
            g0, g1, N = groups[gi]
            inp = self.inputs[gi % 2]
            if self._gfree[gi % 2] is not None:
                rs.wait_event(self._gfree[gi % 2])   # the group before last has been simulated
            if self.group == 1:
                rk, rp_, rsl, rd = keys[t], plens[t], slens[t], dest
            else:
                gk, gp, gs, gd = self.gbuf[gi % 2]
                with torch.cuda.stream(rs):  # stage the interval into the group buffer
                    c = col[t]
                    gk[c:c + n].copy_(keys[t])
                    gp[c:c + n].copy_(plens[t])
                    gs[c:c + n].copy_(slens[t])
                    gd[:len(self.replicas) * N].view(len(self.replicas), N)[:, c:c + n].copy_(dest)
                rk, rp_, rsl = gk[:N], gp[:N], gs[:N]
                rd = gd[:len(self.replicas) * N].view(len(self.replicas), N)
            st_ev = self._event(rs)
            staged.append(st_ev)
            self._dest_free[b] = st_ev if self.group > 1 else None
            if t == g1 - 1:
                for e in staged[:-1]:
                    rs.wait_event(e)                 # the other intervals of the group are staged
                staged = []
                p0 = self._event(rs, True) if mark else None
                replay_partition(rc, self.replay, rk, rp_, rsl, rd, inp)
                parted = self._event(rs, mark)
                if mark:
                    self.part_marks.append((p0, parted))
                if self.group == 1:
                    self._dest_free[b] = parted
                self.ystream.wait_event(parted)
                y0 = self._event(self.ystream, True) if mark else None
                replay_simulate(self.yctx, self.replay, inp, self.ctr)
                replayed = self._event(self.ystream, mark)
                if mark:
                    self.replay_marks.append((y0, replayed))
                self._gfree[gi % 2] = replayed
        for s in self.pstreams + self.rstreams + [self.ystream]:
            self.mstream.wait_event(self._event(s))

    def reset(self):
        """Empty the simulators and counters.  Both are enqueued on the main stream, which
        ``run`` left waiting for all of the pipeline's streams and which the next ``run``
        makes every stream wait for: no host synchronisation is needed."""
        import torch
        self.replay.reset()
        with torch.cuda.stream(self.mstream):
            self.ctr.zero_()
        self._reset_events()

    def sync(self):
        for c in self.contexts:
            c.sync()

    def quiesce(self):
        """Wait for all enqueued work and forget the events that ordered it (e.g. before
        capturing a CUDA graph of ``run``)."""
        self.sync()
        self._reset_events()

    def close(self):
        self.sync()
        for buf in self.plans:
            for pl in buf:
                pl.close()
        self.replay.close()
        for g in self.rings:
            if g is not None:
                g.close()
        for i in self.inputs:
            i.close()
        for c in self.pctxs + self.rctxs + [self.yctx]:
            c.close()
