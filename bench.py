#!/usr/bin/env python
"""Throughput of the planned prefix-affinity routing hot path on GB300.

One step = one pass of the whole hot path over the 70B-shaped primary trace:
for each of its 12 control intervals, hash every request's prefix span, build
the plans from the previous interval's keys, route all 20 (policy, seed)
replicas, and shadow-replay them through the LRU simulators.  Inputs (the
token arenas of all intervals, ~18.6 GB) are resident in HBM before timing
starts and are larger than L2, so no flush is needed between steps.

Prints ONE JSON line (rank 0).  ``--impl reference`` times the CPU oracle (the
plain C restatement of the method) on a bounded sample of the same workload.
Under torchrun with N > 1 each rank runs an independent replica of the
workload (the path needs no exchange between GPUs): value = requests of all
ranks / max time over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "requests/s routed+shadow-replayed on 1 GB300 (and % HBM roofline); plan-build ms"
UNIT = "requests/s"


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="large")
    ap.add_argument("--cpu-sample", type=int, default=262144,
                    help="keys mode: requests of interval 0 in the CPU oracle's timed sample")
    ap.add_argument("--batch", type=int, default=1024)
    ap.add_argument("--sm-split", type=int, default=0,
                    help="run hashing and candidates on all but N SMs and the load-dependent route resolution on "
                         "the other N (green contexts), so that it overlaps the next interval's hashing")
    ap.add_argument("--graph", action=argparse.BooleanOptionalAction, default=None,
                    help="capture the whole step (every interval) once as a CUDA graph and replay it, so that the "
                         "host enqueues one graph per step instead of every launch (default: on for configurations "
                         "whose inputs stay resident, off in keys mode, whose few large intervals the host "
                         "enqueues in a fraction of the step, and with --sm-split or --per-interval); kernel times "
                         "and the roofline then come from one ordinary step after the timed region")
    ap.add_argument("--fresh-plans", action="store_true",
                    help="plan every interval from its own keys (the fresh plan of the replanning study) "
                         "instead of from the previous interval's")
    ap.add_argument("--trace-seed", type=int, default=None,
                    help="seed of the trace realisation (default: the configuration's); ranks add their rank")
    ap.add_argument("--token-lru", action="store_true",
                    help="replay with token-weighted LRU capacities (byte-aware variant)")
    ap.add_argument("--policies", default="",
                    help="comma-separated dispatch policies replacing the configuration's (same seeds), "
                         "e.g. CR,P2C,RR,HASH,CHWBL")
    ap.add_argument("--clocks-out", default="",
                    help="keep the nvidia-smi clock samples of the timed region in this CSV file (default: a "
                         "temporary file, removed after it is summarised)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-overlap", action="store_true", help="build plans in line instead of on a second stream")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--keys-mode", action="store_true",
                    help="hash each interval's arena on its own and time plans + route + replay over resident keys "
                         "(automatic when the arenas do not fit in HBM)")
    ap.add_argument("--per-interval", action="store_true",
                    help="drive one interval at a time (Pipeline) instead of keeping several intervals' plans and "
                         "routes in flight (TracePipeline)")
    ap.add_argument("--depth", type=int, default=16, help="multi-interval driver: intervals in flight")
    ap.add_argument("--plan-streams", type=int, default=8, help="multi-interval driver: streams building plans")
    ap.add_argument("--route-streams", type=int, default=4, help="multi-interval driver: streams routing")
    ap.add_argument("--replay-group", type=int, default=None,
                    help="multi-interval driver: consecutive intervals replayed by one call (default: "
                         "max(2, min(16, 65536 // mean requests per interval)))")
    ap.add_argument("--trace-min-interval", type=int, default=None,
                    help="resident inputs: mean requests per interval from which the multi-interval "
                         "driver runs the trace (default: 0 with a CUDA graph, 65536 without, where many "
                         "small intervals are bound by the host's launch rate)")
    ap.add_argument("--replay-priority", choices=["high", "low"], default="low",
                    help="keys mode: priority of the replay stream (plans get the other one)")
    ap.add_argument("--intervals", type=int, default=0,
                    help="profiling aid: run only the first N intervals (the JSON line says so)")
    args = ap.parse_args(argv)
    args.graph_auto = args.graph is None
    if args.graph is None:
        args.graph = not (args.sm_split or args.per_interval)
    args.trace_min_interval_auto = args.trace_min_interval is None
    if args.trace_min_interval is None:
        args.trace_min_interval = 0 if args.graph else 65536
    return args


def with_policies(cfg, args):
    """The configuration with --policies and --token-lru applied (unchanged without them)."""
    if getattr(args, "token_lru", False):
        cfg = cfg.token_lru()
    if getattr(args, "trace_seed", None) is not None:
        import dataclasses
        cfg = dataclasses.replace(cfg, trace_seed=args.trace_seed)
    if not getattr(args, "policies", ""):
        return cfg
    import dataclasses
    pols = [p.strip() for p in args.policies.split(",") if p.strip()]
    return dataclasses.replace(cfg, policies=pols, name=f"{cfg.name} [{','.join(pols)}]")


def plan_stats(plan_ms):
    """Median and max plan-build time per interval; empty when no replica uses a plan."""
    if plan_ms.size == 0:
        return {"median": None, "max": None, "builds_per_step": 0}
    return {"median": float(np.median(plan_ms)), "max": float(plan_ms.max()),
            "builds_per_step": int(plan_ms.shape[1])}


def isolated_plan_ms(pipe, keys, n_max: int = 8):
    """Plan build timed alone on an otherwise idle device: for intervals 1..n_max, one
    cr_build_plans call (every plan variant the replicas need, from the previous
    interval's keys) between two events on the plan stream; median and max in ms."""
    import torch
    from paper_2608_19677_gb300 import build_plans, plan_params
    if not pipe.plan_keys or len(keys) < 2:
        return {"median": None, "max": None, "intervals": 0}
    torch.cuda.synchronize()
    ps, pc = pipe.pstreams[0], pipe.pctxs[0]
    out = []
    for t in range(1, min(len(keys), n_max + 1)):
        pk = keys[t - 1]
        num, den = pipe.qcap(int(pk.shape[0]))
        params = [plan_params(pipe.R, pipe.W, num, den, v, seed=s, epoch=t) for v, s in pipe.plan_keys]
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(ps)
        build_plans(pc, pk, params, pipe.plans[0])
        e1.record(ps)
        e1.synchronize()
        out.append(e0.elapsed_time(e1))
    pc.sync()
    return {"median": float(np.median(out)), "max": float(np.max(out)), "intervals": len(out),
            "variants_per_build": len(pipe.plan_keys)}


def workload_config(cfg, B, fresh=False):
    return {
        "workload": (f"{cfg.name}: {cfg.R} destinations, {cfg.total_keys} keys Zipf s={cfg.zipf_s}"
                     f"{' (hottest capped)' if cfg.hot_cap else ''}, {cfg.n_requests} requests over "
                     f"{cfg.n_intervals} x {cfg.interval_s:g} s intervals, prefix {cfg.plen}, suffix {cfg.suffix}, "
                     f"{len(cfg.policies)} policies x {len(cfg.seeds)} seeds, LRU caps {cfg.caps}"),
        "requests_per_step": cfg.n_requests,
        "intervals": cfg.n_intervals,
        "destinations": cfg.R,
        "replicas": len(cfg.replicas),
        "policies": cfg.policies,
        "lru_caps": cfg.caps,
        "lru_capacity_unit": "prefix tokens" if cfg.lru_tokens else "prefixes",
        "slots_per_destination": cfg.W,
        "batch_B": B,
        "plans_from": "each interval's own keys (fresh)" if fresh else "the previous interval's keys",
        "rate_drift_sigma": cfg.drift,
        "trace_seed": cfg.trace_seed,
        "l2": "inputs larger than L2 (token arenas of all intervals resident in HBM)",
    }


# ----------------------------------------------------------------- clocks ---
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int, out_path: str = ""):
        self.dev = device_index
        self.proc = None
        self.keep = bool(out_path)  # a caller-chosen file is kept; a temporary one is removed
        if out_path:
            self.path = out_path
        else:
            import tempfile
            fd, self.path = tempfile.mkstemp(prefix=f"cr_clocks_{device_index}_", suffix=".csv")
            os.close(fd)

    def start(self):
        try:
            if os.path.dirname(self.path):
                os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.dev), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not self.keep:
            try:
                os.remove(self.path)
            except OSError:
                pass
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def hash_traffic(alg_bytes_per_launch: float):
    """DRAM bytes per hash launch from the committed ncu capture, scaled by algorithmic
    bytes; None when the kernel source has changed since the capture."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "k_hash_prefixes_traffic.txt")
    src = os.path.join(ROOT, "paper_2608_19677_gb300", "csrc", "cr_hash.cu")
    try:
        kv = {}
        for line in open(path):
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split(None, 1)
                kv[k] = v
        if kv.get("source_sha256") != hashlib.sha256(open(src, "rb").read()).hexdigest():
            return None
        ratio = (float(kv["dram_bytes_read"]) + float(kv["dram_bytes_write"])) / float(kv["algorithmic_bytes"])
        return ratio * alg_bytes_per_launch
    except Exception:
        return None


def lru_traffic(alg_bytes_per_launch: float, pairs_per_launch: float):
    """DRAM bytes per LRU replay launch from the committed ncu capture (bytes per (request,
    replica) pair there, times this launch's pairs); None when the replay source has changed
    since the capture."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "k_lru_stamp_traffic.txt")
    src = os.path.join(ROOT, "paper_2608_19677_gb300", "csrc", "cr_replay.cu")
    try:
        kv = {}
        for line in open(path):
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split(None, 1)
                kv[k] = v
        if kv.get("source_sha256") != hashlib.sha256(open(src, "rb").read()).hexdigest():
            return None
        per_pair = (float(kv["dram_bytes_read"]) + float(kv["dram_bytes_write"])) / float(kv["pairs"])
        return per_pair * pairs_per_launch
    except Exception:
        return None


# ----------------------------------------------------------------- oracle ---
def oracle_interval_step(trace, sample, threads: int, B: int) -> float:
    """One timed pass of the CPU oracle, as it stands, over interval 0 of a resident-arena
    configuration: hash every request (the arena split in `threads` request ranges), the
    plans (from interval 0's own keys), then route and replay every replica; independent
    ranges, plan variants and replicas run on `threads` host threads (each oracle call is
    plain single-threaded C and releases the interpreter lock).  Returns seconds."""
    import concurrent.futures as cf
    import oracle as O
    import oracle.pipeline as OP
    cfg = trace.cfg
    reps = cfg.replicas
    tok, off, iv = sample["tok"], sample["off"], sample["iv"]
    rings = OP.rings_for(cfg)
    n = iv.n
    t0 = time.perf_counter()
    cuts = [n * i // threads for i in range(threads + 1)]

    def hash_range(ab):
        a, b = ab
        return O.hash_prefixes(tok, off[a:b], iv.plen[a:b]) if b > a else np.zeros(0, np.uint64)

    with cf.ThreadPoolExecutor(threads) as ex:
        keys = np.concatenate(list(ex.map(hash_range, zip(cuts[:-1], cuts[1:]))))
    num, den = trace.qcap(n)
    variants = sorted({(OP.VARIANT_OF[p], sd if OP.VARIANT_OF[p] == "RANDOM" else 0)
                       for p, sd in reps if p in OP.VARIANT_OF})

    def build(vs):
        v, sd = vs
        return vs, O.build_plan(keys, cfg.R, cfg.W, num, den, variant=v, seed=sd, epoch=0)

    with cf.ThreadPoolExecutor(threads) as ex:
        built = dict(ex.map(build, variants))

    def one(i):
        p, sd = reps[i]
        v = OP.VARIANT_OF.get(p)
        plan = built[(v, sd if v == "RANDOM" else 0)] if v is not None else None
        d, _ = O.route([plan], [OP.ROUTE_AS.get(p, p)], [sd], cfg.R, keys, iv.g0, B, rings=[rings[i]])
        rp = O.Replay(1, cfg.R, cfg.caps, tokens=cfg.lru_tokens)
        rp.step(keys, iv.plen, iv.slen, d)
        return int(rp.ctr[..., 0].sum())

    with cf.ThreadPoolExecutor(threads) as ex:
        done = list(ex.map(one, range(len(reps))))
    assert all(x == n * len(cfg.caps) for x in done)
    return time.perf_counter() - t0


def oracle_interval_sample(trace):
    """Input preparation (untimed): interval 0's token arena on the host."""
    import tracegen as tg
    iv = trace.interval(0)
    tok, off = tg.arena_host(trace, iv, 4)
    return {"tok": tok, "off": off, "iv": iv, "n": iv.n}


def token_bytes(trace) -> float:
    """Bytes of the token arenas of every interval of the trace."""
    cfg = trace.cfg
    rec_tokens = float(trace.key_plen.astype(np.float64).mean()) + cfg.suffix + 3
    return 4.0 * rec_tokens * float(sum(trace.counts[:cfg.n_intervals]))


def auto_schedule(args, trace):
    """Defaults that depend on the interval size (mean requests per interval, m): a CUDA
    graph of the step when m < 262,144 (many intervals, each too short to hide the host's
    launches; the Large sweep's ~1M-request intervals run better without one), and
    max(2, min(16, 65536 // m)) consecutive intervals per replay call (the replay is the
    one serial chain; grouping short intervals shortens it)."""
    cfg = trace.cfg
    m = sum(int(c) for c in trace.counts[:cfg.n_intervals]) / max(cfg.n_intervals, 1)
    if args.graph_auto:
        args.graph = bool(m < 262144 and not (args.sm_split or args.per_interval))
        if args.trace_min_interval_auto:
            args.trace_min_interval = 0 if args.graph else 65536
    if args.replay_group is None:
        args.replay_group = int(max(2, min(16, 65536 // max(int(m), 1))))


def keys_mode_for(args, trace, free_bytes: float = 280e9) -> bool:
    """Keys mode when asked, or when the arenas would not fit in (60% of) free device memory."""
    return bool(args.keys_mode) or token_bytes(trace) > 0.6 * free_bytes


def oracle_keys_sample(trace, S: int):
    """Input preparation for the keys-mode oracle baseline (untimed): the first S requests of
    interval 0 with their routing keys, hashed by the oracle from the prefix tokens (each
    distinct key's prefix once, since requests that carry a key share its prefix)."""
    import oracle as O
    import tracegen as tg
    iv = trace.interval(0)
    S = min(S, iv.n)
    kid = iv.key_id[:S]
    ids = np.unique(kid)
    keys = np.empty(S, np.uint64)
    kv = np.empty(ids.size, np.uint64)
    chunk = 50000
    for a in range(0, ids.size, chunk):
        tok, off, pl = tg.prefix_spans(trace, ids[a:a + chunk])
        kv[a:a + chunk] = O.hash_prefixes(tok, off, pl)
    keys[:] = kv[np.searchsorted(ids, kid)]
    return {"keys": keys, "plen": iv.plen[:S].copy(), "slen": iv.slen[:S].copy(), "g0": iv.g0, "n": S,
            "of": iv.n}


def oracle_keys_step(trace, sample, threads: int, B: int) -> float:
    """One timed pass of the CPU oracle, as it stands, over a keys-mode sample: the plans of
    interval 0 (from its own keys), then routing and replay of every replica; independent plan
    variants and replicas run on `threads` host threads (each oracle call is plain
    single-threaded C and releases the interpreter lock).  Returns seconds."""
    import concurrent.futures as cf
    import oracle as O
    import oracle.pipeline as OP
    cfg = trace.cfg
    reps = cfg.replicas
    keys, plen, slen = sample["keys"], sample["plen"], sample["slen"]
    rings = OP.rings_for(cfg)
    num, den = trace.qcap(sample["n"])
    variants = sorted({(OP.VARIANT_OF[p], s if OP.VARIANT_OF[p] == "RANDOM" else 0)
                       for p, s in reps if p in OP.VARIANT_OF})
    t0 = time.perf_counter()

    def build(vs):
        v, sd = vs
        return vs, O.build_plan(keys, cfg.R, cfg.W, num, den, variant=v, seed=sd, epoch=0)

    with cf.ThreadPoolExecutor(threads) as ex:
        built = dict(ex.map(build, variants))

    def one(i):
        p, sd = reps[i]
        v = OP.VARIANT_OF.get(p)
        plan = built[(v, sd if v == "RANDOM" else 0)] if v is not None else None
        d, _ = O.route([plan], [OP.ROUTE_AS.get(p, p)], [sd], cfg.R, keys, sample["g0"], B, rings=[rings[i]])
        rp = O.Replay(1, cfg.R, cfg.caps, tokens=cfg.lru_tokens)
        rp.step(keys, plen, slen, d)
        return int(rp.ctr[..., 0].sum())

    with cf.ThreadPoolExecutor(threads) as ex:
        done = list(ex.map(one, range(len(reps))))
    assert all(x == sample["n"] * len(cfg.caps) for x in done)
    return time.perf_counter() - t0


def keys_sample_text(cfg, sample, threads):
    return (f"first {sample['n']} of the {sample['of']} requests of interval 0 (of {cfg.n_intervals}), all "
            f"{len(cfg.replicas)} replicas x {len(cfg.caps)} capacities: plans from their keys + route + replay, "
            f"keys hashed beforehand (the device step also starts from resident keys); C oracle, "
            f"{threads} host thread(s) over independent plan variants and replicas")


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import tracegen as tg
    cfg = with_policies(tg.CONFIGS[args.config], args)
    trace = tg.Trace(cfg)
    if keys_mode_for(args, trace):
        return run_reference_keys(args, cfg, trace)
    threads = os.cpu_count() or 1
    sample = oracle_interval_sample(trace)
    for _ in range(args.warmup):
        oracle_interval_step(trace, sample, threads, args.batch)
    each = [oracle_interval_step(trace, sample, threads, args.batch) for _ in range(args.steps)]
    dt = float(np.mean(each)) if each else 0.0
    value = sample["n"] / dt if dt > 0 else 0.0
    text = (f"interval 0 of {cfg.n_intervals} ({sample['n']} requests, all {len(cfg.replicas)} replicas) per step, "
            f"hash+plan+route+replay, C oracle on {threads} host threads over request ranges, plan variants and "
            f"replicas")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
            "config": workload_config(cfg, args.batch, args.fresh_plans),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": text},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_reference_keys(args, cfg, trace):
    """Reference arm of a keys-mode configuration: each step is one oracle pass over the
    bounded sample, on all host cores."""
    threads = os.cpu_count() or 1
    sample = oracle_keys_sample(trace, args.cpu_sample)
    for _ in range(args.warmup):
        oracle_keys_step(trace, sample, threads, args.batch)
    each = [oracle_keys_step(trace, sample, threads, args.batch) for _ in range(args.steps)]
    dt = float(np.mean(each)) if each else 0.0
    value = sample["n"] / dt if dt > 0 else 0.0
    cb = {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
          "sample": keys_sample_text(cfg, sample, threads)}
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
            "config": workload_config(cfg, args.batch, args.fresh_plans), "cpu_baseline": cb,
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------- multi-rank ---
# One process per GPU, each running an independent replica of the workload
# (the path has no exchange step, so ranks share nothing but the timing).
def replica_cfg(cfg, rank: int, world: int):
    """The workload of one rank: the same configuration with its own trace seed."""
    import dataclasses
    return dataclasses.replace(cfg, trace_seed=cfg.trace_seed + rank) if world > 1 else cfg


def max_over_ranks(x: float, world: int, device) -> float:
    """The slowest rank's value (the job ends when the last rank does)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank: int, world: int, ms_max: float) -> float:
    """Units of all ranks per second of the slowest rank's time."""
    return units_per_rank * world / (ms_max / 1e3)


def close_in_order(pipe, ctx, part):
    """With an SM partition, free what uses its streams before the partition itself: the
    pipeline (plans, replay, rings, its own contexts), then the context on the big stream."""
    if part is None:
        return
    pipe.close()
    ctx.close()
    part.close()


# ----------------------------------------------------------------- ours ---
def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    import torch
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.gpus > 1 and world == 1:
        sys.exit("--gpus > 1 must be launched with torch.distributed.run (one process per GPU)")
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if world > 1:
            dist.barrier()

    import __graft_entry__
    if rank == 0 or world == 1:
        __graft_entry__.build()
    barrier()
    import paper_2608_19677_gb300 as P
    import tracegen as tg
    from paper_2608_19677_gb300.pipeline import Pipeline

    cfg = with_policies(tg.CONFIGS[args.config], args)
    cfg = replica_cfg(cfg, rank, world)  # independent replica per rank
    trace = tg.Trace(cfg)
    if args.intervals:
        import dataclasses
        cfg = dataclasses.replace(cfg, n_intervals=args.intervals, name=f"{cfg.name} (first {args.intervals} "
                                  f"intervals only)", n_requests=int(sum(trace.counts[:args.intervals])))
        trace.cfg = cfg
    auto_schedule(args, trace)
    dev = torch.device("cuda", local)
    part = None
    if args.sm_split and args.graph:
        sys.exit("--sm-split and --graph cannot be combined (a graph capture would span the partition's "
                 "streams and the resolve-stream switch)")
    if args.sm_split:  # main stream on the large SM partition, route resolution on the small one
        part = P.Partition(local, args.sm_split)
        torch.cuda.set_stream(part.big)
    elif args.graph:  # graphs are captured on a stream of their own; torch's ops follow it
        torch.cuda.set_stream(torch.cuda.Stream(dev))
    stream = torch.cuda.current_stream(dev)
    resolve_stream = part.small if part is not None else None

    # keys mode: when the token arenas of all intervals do not fit in HBM (the
    # large configuration holds ~600 GB of tokens), every interval's arena is
    # generated and hashed one at a time (each hash launch timed on its own),
    # and the timed steps run plans + route + replay over the resident keys.
    free, _total = torch.cuda.mem_get_info(dev)
    if keys_mode_for(args, trace, float(free)):
        return run_keys_mode(args, cfg, trace, dev, stream, world, rank, barrier, resolve_stream, part)

    # inputs resident in HBM (generated on the device, untimed)
    inputs = []
    hash_bytes = []
    for t in range(cfg.n_intervals):
        iv = trace.interval(t)
        tok, off = tg.arena_device(trace, iv, 4, device=dev)
        plen = torch.from_numpy(iv.plen.view(np.int32)).to(dev)
        slen = torch.from_numpy(iv.slen.view(np.int32)).to(dev)
        inputs.append((t, tok, off, plen, slen, iv.g0, iv.n))
        # algorithmic bytes of one hash launch: 4 P + 8 (offset) + 4 (length) + 8 (key) per request
        hash_bytes.append(4 * int(iv.plen.astype(np.int64).sum()) + 20 * iv.n)
    torch.cuda.synchronize()
    n_step = sum(x[6] for x in inputs)
    max_n = max(x[6] for x in inputs)
    # several intervals in flight pay off when intervals are large; many small intervals are
    # bound by launches from the host, which the one-interval driver issues fewer of
    big = n_step / max(cfg.n_intervals, 1) >= args.trace_min_interval
    if big and not (args.per_interval or part is not None or cfg.drift or args.no_overlap):
        return run_resident_trace(args, cfg, trace, inputs, hash_bytes, dev, stream, world, rank, barrier)

    ctx = P.Context(local, stream)
    pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, trace.qcap, batch_B=args.batch, max_n=max_n,
                    overlap=not args.no_overlap, vnodes=cfg.vnodes, fresh=args.fresh_plans,
                    lru_tokens=cfg.lru_tokens, resolve_stream=resolve_stream)
    marks = [[[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(cfg.n_intervals)]
             for _ in range(max(args.steps, 1))]

    plan_marks = [[] for _ in range(max(args.steps, 1))]

    hash_marks = [[] for _ in range(max(args.steps, 1))]
    route_marks = [[] for _ in range(max(args.steps, 1))]
    replay_marks = [[] for _ in range(max(args.steps, 1))]

    def step(k=None):
        pipe.reset()
        for i, (t, tok, off, plen, slen, g0, n) in enumerate(inputs):
            pipe.interval(t, tok, off, plen, slen, g0, marks=marks[k][i] if k is not None else None,
                          plan_next=i + 1 < len(inputs))
        pipe.finish()
        if k is not None:
            plan_marks[k] = list(pipe.plan_marks)
            hash_marks[k] = list(pipe.hash_marks)
            route_marks[k] = list(pipe.route_marks)
            replay_marks[k] = list(pipe.replay_marks)

    def launches():
        return pipe.launches

    for _ in range(max(args.warmup, 1 if args.graph else 0)):  # a graph captures warm buffers only
        step()
    ctx.sync()
    torch.cuda.synchronize()

    # ---- optional CUDA graph of the whole step ---------------------------------
    graph, graph_launches = None, 0
    if args.graph:
        pipe.quiesce()
        graph = torch.cuda.CUDAGraph()
        lc0 = launches()
        with torch.cuda.graph(graph, stream=stream):
            step()
        graph_launches = launches() - lc0  # library launches in one replay
        graph.replay()
        torch.cuda.synchronize()

    # ---- timed region: K steps, stage events on the launching stream -------
    clocks = ClockSampler(local, args.clocks_out)
    clocks.start()
    time.sleep(0.3)
    barrier()
    torch.cuda.synchronize()
    l0 = launches()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for k in range(args.steps):
        if graph is not None:
            graph.replay()
        else:
            step(k)
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    n_launch = graph_launches * args.steps if graph is not None else launches() - l0
    clk = clocks.stop()
    if graph is not None:
        # per-stage times and the hash roofline from one ordinary step after the timed region
        pipe.quiesce()
        step(0)
        torch.cuda.synchronize()
    marked = [0] if graph is not None else list(range(args.steps))
    stage_ms = np.zeros((len(marked), cfg.n_intervals, 4))
    for j, k in enumerate(marked):
        for i in range(cfg.n_intervals):
            m = marks[k][i]
            for s in range(4):
                stage_ms[j, i, s] = m[s].elapsed_time(m[s + 1])
    hash_marks, plan_marks = [hash_marks[k] for k in marked], [plan_marks[k] for k in marked]
    route_marks, replay_marks = [route_marks[k] for k in marked], [replay_marks[k] for k in marked]
    ctx.sync()
    ms_total = ev0.elapsed_time(ev1)
    ms = ms_total / args.steps
    ms_max = max_over_ranks(ms, world, dev)
    value = job_throughput(n_step, world, ms_max)

    # per-stage summaries (hash and plan builds are timed on their own streams)
    hash_ms = np.array([[a.elapsed_time(b) for a, b in hm] for hm in hash_marks])
    plan_wait_ms = stage_ms[:, :, 0] + stage_ms[:, :, 1]
    plan_ms = np.array([[a.elapsed_time(b) for a, b in pm] for pm in plan_marks])
    # route and replay calls timed on their own streams, after their waits
    route_ms = np.array([[a.elapsed_time(b) for a, b in rm] for rm in route_marks])
    replay_ms = np.array([[a.elapsed_time(b) for a, b in ym] for ym in replay_marks])
    hb = np.array(hash_bytes, dtype=np.float64)
    hash_gbs = float((hb[None, :] / (hash_ms / 1e3)).mean() / 1e9)
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    peak_src = "measured" if "hbm_gbs" in peaks else "fallback"
    traffic = hash_traffic(float(hb.mean()))
    roofline = {"kernel": "k_hash_prefixes", "bound": "hbm", "achieved": hash_gbs, "peak": hbm_peak,
                "peak_source": peak_src, "unit": "GB/s", "frac": hash_gbs / hbm_peak, "traffic": traffic,
                "algorithmic_bytes_per_launch_mean": float(hb.mean()),
                "avg_launch_ms": float(hash_ms.mean())}
    rr_ms = float((route_ms + replay_ms).sum(axis=1).mean())
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": dict(workload_config(cfg, args.batch, args.fresh_plans), sm_split=args.sm_split or None),
        "roofline": roofline,
        "stages_ms_per_step": {"hash": float(hash_ms.sum(1).mean()),
                               "main_wait_for_keys_and_plans": float(plan_wait_ms.sum(1).mean()),
                               "route": float(route_ms.sum(1).mean()), "replay": float(replay_ms.sum(1).mean())},
        "plan_build_ms": dict(plan_stats(plan_ms),
                              per="interval (histogram + admission + placement + table for all plan variants), "
                                  + ("on its own stream, overlapped with hash/route/replay" if pipe.overlap
                                     else "in line on the main stream")),
        "streams": ("hash (low priority) / planner (high priority) / route+replay: overlapped"
                    if pipe.overlap else "one stream"),
        "route_replay_requests_per_s": n_step / (rr_ms / 1e3),
        "route_replay_note": "requests over the summed route and replay call times; the calls overlap hashing, "
                             "planning and each other",
        "gpu_launches": int(n_launch),
        "clocks": clk,
    }
    if graph is not None:
        line["cuda_graph"] = ("the timed steps replay one CUDA graph of the whole step; stage times, plan-build "
                              "times and the roofline come from one ordinary step after the timed region")
        pipe.quiesce()

    # ---- replanning under drift (untimed study) ----------------------------
    if cfg.drift:
        line["replan"] = replan_study(args, ctx, cfg, trace, inputs, dev, stream, max_n)
    # ---- end to end through the public API with pinned host buffers -------
    if not args.no_e2e:
        line["e2e"] = e2e(args, ctx, pipe, inputs, dev, stream, n_step, world)
    # ---- CPU baseline (rank 0, N = 1) ---------------------------------------
    if not args.no_cpu_baseline and world == 1:
        sample = oracle_interval_sample(trace)
        nproc = os.cpu_count() or 1
        t1 = oracle_interval_step(trace, sample, 1, args.batch)
        tn = oracle_interval_step(trace, sample, nproc, args.batch)
        line["cpu_baseline"] = {"value": sample["n"] / tn, "unit": UNIT, "cores": nproc, "kind": "oracle",
                                "sample": f"interval 0 of {cfg.n_intervals} ({sample['n']} requests, all "
                                          f"{len(cfg.replicas)} replicas), hash+plan+route+replay, C oracle on "
                                          f"{nproc} host threads over request ranges, plan variants and replicas",
                                "single_thread": {"value": sample["n"] / t1, "unit": UNIT, "cores": 1},
                                "nproc": nproc}
    if rank == 0:
        print(json.dumps(line), flush=True)
    close_in_order(pipe, ctx, part)
    if world > 1:
        dist.destroy_process_group()


def replan_study(args, ctx, cfg, trace, inputs, dev, stream, max_n):
    """Replanning under drift, after the timed region (supplement "Replanning Under Drift"):
    cache and count churn between the fresh LPT plans of consecutive intervals (cr_plan_diff,
    timed with CUDA events), and per-interval LRU hit rates when every interval is routed with a
    stale plan (previous interval's keys) or a fresh one (its own keys)."""
    import torch
    import paper_2608_19677_gb300 as P
    from paper_2608_19677_gb300.pipeline import Pipeline
    keys = []
    for (t, tok, off, plen, slen, g0, n) in inputs:
        k = torch.empty(n, dtype=torch.int64, device=dev)
        P.hash_prefixes(ctx, tok, off, plen, 0, out=k)
        keys.append(k)
    plans = []
    for t, k in enumerate(keys):
        num, den = trace.qcap(int(k.shape[0]))
        plans.append(P.build_plan(ctx, k, P.plan_params(cfg.R, cfg.W, num, den, "LPT", epoch=t)))
    ctx.sync()
    transitions, diff_ms = [], []
    for t in range(len(plans) - 1):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        d = P.plan_diff(ctx, plans[t], plans[t + 1])  # blocking
        e1.record(stream)
        e1.synchronize()
        diff_ms.append(e0.elapsed_time(e1))
        cache, count = P.churn(d)
        transitions.append(dict(transition=f"{t}->{t + 1}", cache_churn=cache, count_churn=count, **d))
    pols = sorted(set(cfg.policies), key=cfg.policies.index)
    rows = {p: [i for i, (q, _) in enumerate(cfg.replicas) if q == p] for p in pols}

    def hit_rates(fresh):
        pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, trace.qcap, batch_B=args.batch, max_n=max_n,
                        overlap=not args.no_overlap, vnodes=cfg.vnodes, fresh=fresh,
                        lru_tokens=cfg.lru_tokens)
        pipe.reset()
        prev = torch.zeros_like(pipe.ctr)
        out = {p: [] for p in pols}
        for i, (t, tok, off, plen, slen, g0, n) in enumerate(inputs):
            pipe.interval(t, None, off, plen, slen, g0, plan_next=i + 1 < len(inputs), keys=keys[i])
            pipe.finish()
            pipe.sync()
            cur = pipe.ctr.clone()
            dt = (cur - prev)[:, 0]  # first LRU capacity
            prev = cur
            for p in pols:
                req = int(dt[rows[p], :, 0].sum())
                out[p].append(int(dt[rows[p], :, 1].sum()) / req if req else 0.0)
        return out

    stale, fresh = hit_rates(False), hit_rates(True)
    return {
        "sigma": cfg.drift,
        "transitions": transitions,
        "plan_diff_ms": {"median": float(np.median(diff_ms)), "max": float(np.max(diff_ms)),
                         "per": "cr_plan_diff call (blocking: kernels + counter read-back)"},
        "hit_rate_per_interval": {"stale_plan": stale, "fresh_plan": fresh,
                                  "lru_capacity": cfg.caps[0]},
        "kv_loss_points_of_stale": {p: [100.0 * (fresh[p][t] - stale[p][t]) for t in range(1, len(inputs))]
                                    for p in pols},
        "note": "fresh = plan from the interval's own keys; stale = plan from the previous interval's keys "
                "(the pipeline's default); LRU state carries over intervals, so a fresh plan's hit rate "
                "includes its rewarming misses",
    }


def run_keys_mode(args, cfg, trace, dev, stream, world, rank, barrier, resolve_stream=None, part=None):
    import torch
    import torch.distributed as dist
    import paper_2608_19677_gb300 as P
    import tracegen as tg
    from paper_2608_19677_gb300.pipeline import Pipeline, TracePipeline

    ctx = P.Context(dev.index if dev.index is not None else 0, stream)
    keys, plens, slens, g0s, ns = [], [], [], [], []
    hash_ms, hash_bytes = [], []
    for t in range(cfg.n_intervals):
        iv = trace.interval(t)
        tok, off = tg.arena_device(trace, iv, 4, device=dev)
        plen = torch.from_numpy(iv.plen.view(np.int32)).to(dev)
        k = torch.empty(iv.n, dtype=torch.int64, device=dev)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        P.hash_prefixes(ctx, tok, off, plen, 0, out=k)
        e1.record(stream)
        e1.synchronize()
        hash_ms.append(e0.elapsed_time(e1))
        hash_bytes.append(4 * int(iv.plen.astype(np.int64).sum()) + 20 * iv.n)
        keys.append(k)
        plens.append(plen)
        slens.append(torch.from_numpy(iv.slen.view(np.int32)).to(dev))
        g0s.append(iv.g0)
        ns.append(iv.n)
        del tok, off
    torch.cuda.synchronize()
    torch.cuda.empty_cache()  # the arenas are gone: only keys and lengths stay on the device
    n_step = sum(ns)
    trace_mode = not args.per_interval and resolve_stream is None
    if trace_mode:
        pipe = TracePipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, trace.qcap, max_n=max(ns),
                             batch_B=args.batch, depth=args.depth, plan_streams=args.plan_streams,
                             route_streams=args.route_streams, vnodes=cfg.vnodes, fresh=args.fresh_plans,
                             lru_tokens=cfg.lru_tokens, replay_first=args.replay_priority == "high",
                             replay_group=args.replay_group)
    else:
        pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, trace.qcap, batch_B=args.batch, max_n=max(ns),
                        overlap=not args.no_overlap, vnodes=cfg.vnodes, fresh=args.fresh_plans,
                        lru_tokens=cfg.lru_tokens, resolve_stream=resolve_stream)
    marks = [[[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(cfg.n_intervals)]
             for _ in range(max(args.steps, 1))]
    plan_marks = [[] for _ in range(max(args.steps, 1))]
    route_marks = [[] for _ in range(max(args.steps, 1))]
    replay_marks = [[] for _ in range(max(args.steps, 1))]

    def step(k=None):
        pipe.reset()
        if trace_mode:
            pipe.run(keys, plens, slens, g0s, mark=k is not None)
        else:
            for t in range(cfg.n_intervals):
                pipe.interval(t, None, None, plens[t], slens[t], g0s[t],
                              marks=marks[k][t] if k is not None else None,
                              plan_next=t + 1 < cfg.n_intervals, keys=keys[t])
            pipe.finish()
        if k is not None:
            plan_marks[k] = list(pipe.plan_marks)
            route_marks[k] = list(pipe.route_marks)
            replay_marks[k] = list(pipe.replay_marks)

    for _ in range(max(args.warmup, 1 if args.graph else 0)):  # a graph captures warm buffers only
        step()
    pipe.sync()
    graph, graph_launches = None, 0
    if args.graph:
        pipe.quiesce()
        graph = torch.cuda.CUDAGraph()
        lc0 = pipe.launches
        with torch.cuda.graph(graph, stream=stream):
            step()
        graph_launches = pipe.launches - lc0
        graph.replay()
        torch.cuda.synchronize()
    # per-launch CUDA events around the library's main kernels, on the streams they run on
    # (graphs: from one ordinary step after the timed region)
    prof_ctxs = pipe.contexts
    for c in prof_ctxs:
        c.profile_enable(0 if graph is not None else 16 * cfg.n_intervals * max(args.steps, 1) + 64)
    clocks = ClockSampler(dev.index or 0, args.clocks_out)
    clocks.start()
    time.sleep(0.3)
    barrier()
    torch.cuda.synchronize()
    l0 = pipe.launches
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for k in range(args.steps):
        if graph is not None:
            graph.replay()
        else:
            step(k)
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    n_launch = graph_launches * args.steps if graph is not None else pipe.launches - l0
    clk = clocks.stop()
    if graph is not None:  # stage and plan times from one ordinary step after the timed region
        pipe.quiesce()
        for c in prof_ctxs:
            c.profile_enable(16 * cfg.n_intervals + 64)
        step(0)
    pipe.sync()
    kern = {}
    for tag in ("plan", "route_cand", "route_resolve", "partition", "replay"):
        n_, ms_ = 0, 0.0
        for c in prof_ctxs:
            a, b = c.profile_read(tag)
            n_, ms_ = n_ + a, ms_ + b
        kern[tag] = {"launches": n_, "avg_ms": ms_ / n_ if n_ else None}
    for c in prof_ctxs:
        c.profile_enable(0)
    ms = ev0.elapsed_time(ev1) / args.steps
    ms_max = max_over_ranks(ms, world, dev)
    marked = [0] if graph is not None else list(range(args.steps))
    plan_marks = [plan_marks[k] for k in marked]
    route_marks, replay_marks = [route_marks[k] for k in marked], [replay_marks[k] for k in marked]
    stage = np.zeros((len(marked), cfg.n_intervals, 4))
    if not trace_mode:
        for j, k in enumerate(marked):
            for t in range(cfg.n_intervals):
                m = marks[k][t]
                for s_ in range(4):
                    stage[j, t, s_] = m[s_].elapsed_time(m[s_ + 1])
    plan_ms = np.array([[a.elapsed_time(b) for a, b in pm] for pm in plan_marks])
    # route and replay calls timed on their own streams, after their waits
    route_ms = float(np.array([[a.elapsed_time(b) for a, b in rm] for rm in route_marks]).sum(1).mean())
    replay_ms = float(np.array([[a.elapsed_time(b) for a, b in ym] for ym in replay_marks]).sum(1).mean())
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    hb = np.array(hash_bytes, dtype=np.float64)
    hms = np.array(hash_ms)
    hash_gbs = float((hb / (hms / 1e3)).mean() / 1e9)
    reps, ncaps = len(cfg.replicas), len(cfg.caps)
    # route + replay algorithmic bytes per request, counted per row: route 8 (key)
    # + 2 per replica (destination); partition 2 read + 4 written per replica;
    # replay 4 + 8 + 8 read per (replica, capacity)
    rr_bytes = 8 + 2 * reps + 6 * reps + 20 * reps * ncaps
    # the timed step is plans + route + replay with nothing else: its throughput is
    # route + replay's (plans overlap them on their own stream)
    rr_rps = n_step / (ms_max / 1e3)
    rr_gbs = rr_bytes * rr_rps / 1e9
    # the dominant kernel of the step: the LRU simulation (a9), one launch per interval; its
    # algorithmic bytes per launch are 20 per (request, replica, capacity): the replay's algorithmic count
    steps_profiled = 1 if graph is not None else args.steps
    req_per_launch = n_step * steps_profiled / max(kern["replay"]["launches"], 1)
    a9_bytes = 20.0 * reps * ncaps * req_per_launch
    lru_ms = kern["replay"]["avg_ms"]
    lru_gbs = a9_bytes / (lru_ms / 1e3) / 1e9 if lru_ms else None
    line = {
        "metric": METRIC, "value": job_throughput(n_step, world, ms_max), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": dict(workload_config(cfg, args.batch, args.fresh_plans), sm_split=args.sm_split or None,
                       step="plans + route + replay over resident keys (the token arenas of all intervals do "
                            "not fit in HBM: each interval's arena was generated and hashed one at a time, each "
                            "hash launch timed alone)",
                       schedule=(f"{args.depth} intervals in flight: plans on {args.plan_streams} streams, routes "
                                 f"on {args.route_streams} streams, the replay in interval order on one stream, "
                                 f"{args.replay_group} intervals per replay call"
                                 if trace_mode else "one interval at a time (plans of the next interval overlap)"),
                       l2="inputs larger than L2 (keys, prefix and suffix lengths of all intervals resident)"),
        "roofline": {"kernel": "k_lru_stamp (a9 LRU replay)", "bound": "hbm", "achieved": lru_gbs,
                     "peak": hbm_peak, "peak_source": "measured" if "hbm_gbs" in peaks else "fallback",
                     "unit": "GB/s", "frac": lru_gbs / hbm_peak if lru_gbs else None,
                     "traffic": lru_traffic(a9_bytes, reps * req_per_launch),
                     "requests_per_launch": req_per_launch,
                     "algorithmic_bytes_per_launch_mean": a9_bytes, "avg_launch_ms": lru_ms,
                     "launches_timed": kern["replay"]["launches"],
                     "note": "20 B per (request, replica, capacity), the algorithmic bytes of the replay step; the kernel reads "
                             "one 16 B record per (request, replica) and decides every capacity from it; the "
                             "kernel is bound by the latency of its per-step dependence chain, not by bytes"},
        "hash_roofline": {"kernel": "k_hash_prefixes", "bound": "hbm", "achieved": hash_gbs, "peak": hbm_peak,
                          "unit": "GB/s", "frac": hash_gbs / hbm_peak, "traffic": hash_traffic(float(hb.mean())),
                          "algorithmic_bytes_per_launch_mean": float(hb.mean()), "avg_launch_ms": float(hms.mean()),
                          "note": "keys mode: each interval's hash timed alone before the timed step"},
        "kernels_ms_per_launch": kern,
        "route_replay": {"requests_per_s": rr_rps, "route_call_ms_per_step": route_ms,
                         "replay_call_ms_per_step": replay_ms,
                         "note": "route and replay run overlapped on two streams; call times are under contention",
                         "algorithmic_bytes_per_request": rr_bytes,
                         "achieved_GBps": rr_gbs, "hbm_frac": rr_gbs / hbm_peak},
        "hash_ms_per_pass": float(hms.sum()),
        "plan_build_ms": dict(plan_stats(plan_ms), note="in the step, under contention with routes and replay",
                              isolated=isolated_plan_ms(pipe, keys) if trace_mode else None),
        "main_wait_for_plans_ms_per_step": float((stage[:, :, 0] + stage[:, :, 1]).sum(1).mean()),
        "gpu_launches": int(n_launch), "clocks": clk,
    }
    if graph is not None:
        line["cuda_graph"] = ("the timed steps replay one CUDA graph of the whole step; stage, route, replay "
                              "and plan-build times come from one ordinary step after the timed region")
    # ---- end to end through the public API with pinned host buffers -------
    if not args.no_e2e and trace_mode:
        line["e2e"] = e2e_keys(args, pipe, keys, plens, slens, g0s, dev, stream, n_step, world)
    # ---- CPU baseline (rank 0, N = 1): the oracle on a bounded sample -------
    if not args.no_cpu_baseline and world == 1:
        sample = oracle_keys_sample(trace, args.cpu_sample)
        nproc = os.cpu_count() or 1
        t1 = oracle_keys_step(trace, sample, 1, args.batch)
        tn = oracle_keys_step(trace, sample, nproc, args.batch)
        line["cpu_baseline"] = {"value": sample["n"] / tn, "unit": UNIT, "cores": nproc, "kind": "oracle",
                                "sample": keys_sample_text(cfg, sample, nproc),
                                "single_thread": {"value": sample["n"] / t1, "unit": UNIT, "cores": 1},
                                "nproc": nproc}
    if rank == 0:
        print(json.dumps(line), flush=True)
    close_in_order(pipe, ctx, part)
    if world > 1:
        dist.destroy_process_group()


def e2e_keys(args, pipe, keys, plens, slens, g0s, dev, stream, n_step, world):
    """Keys mode end to end through the public API: every step copies each interval's keys,
    prefix and suffix lengths from pinned host memory (a copy stream, one event per
    interval, so routing of interval t starts once its inputs have landed), runs the whole
    trace and reads the counters back."""
    import torch
    host = []
    for k, pl, sl in zip(keys, plens, slens):
        h = []
        for x in (k, pl, sl):
            p = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
            p.copy_(x)
            h.append(p)
        host.append(h)
    h2d = sum(x.numel() * x.element_size() for h in host for x in h)
    dbuf = [[torch.empty_like(x, device=dev) for x in h] for h in host]
    copy_stream = torch.cuda.Stream(dev)
    out = torch.empty(pipe.ctr.shape, dtype=torch.int64, pin_memory=True)
    d2h = out.numel() * out.element_size()

    def step():
        pipe.reset()
        start = torch.cuda.Event()
        start.record(stream)
        copy_stream.wait_event(start)  # the previous step's readers are done with the buffers
        ready = []
        with torch.cuda.stream(copy_stream):
            for h, d in zip(host, dbuf):
                for a, b in zip(h, d):
                    b.copy_(a, non_blocking=True)
                e = torch.cuda.Event()
                e.record(copy_stream)
                ready.append(e)
        pipe.run([d[0] for d in dbuf], [d[1] for d in dbuf], [d[2] for d in dbuf], g0s, ready=ready)
        out.copy_(pipe.ctr, non_blocking=True)

    for _ in range(2):
        step()
    torch.cuda.synchronize()
    each = []
    for _ in range(args.e2e_steps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)  # after the counters' read-back on this stream
        e1.synchronize()
        each.append(e0.elapsed_time(e1))
    ms = max_over_ranks(float(np.median(each)), world, dev)
    return {"value": job_throughput(n_step, world, ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "ms_per_step_each": [round(x, 2) for x in each],
            "note": "keys, prefix and suffix lengths of every interval copied from pinned host memory on a copy "
                    "stream each step (routing of an interval waits for its copy), counters read back; median "
                    "of the timed steps"}


def run_resident_trace(args, cfg, trace, inputs, hash_bytes, dev, stream, world, rank, barrier):
    """Resident-arena configurations with the multi-interval driver: every interval's prefix
    spans are hashed on a stream of their own (one event per interval), and TracePipeline
    plans and routes each interval as soon as its keys (and the previous interval's) exist,
    the replay following in interval order."""
    import torch
    import torch.distributed as dist
    import paper_2608_19677_gb300 as P
    from paper_2608_19677_gb300.pipeline import TracePipeline

    ctx = P.Context(dev.index if dev.index is not None else 0, stream)
    n_step = sum(x[6] for x in inputs)
    max_n = max(x[6] for x in inputs)
    pipe = TracePipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, trace.qcap, max_n=max_n, batch_B=args.batch,
                         depth=args.depth, plan_streams=args.plan_streams, route_streams=args.route_streams,
                         vnodes=cfg.vnodes, fresh=args.fresh_plans, lru_tokens=cfg.lru_tokens,
                         replay_first=args.replay_priority == "high", replay_group=args.replay_group)
    hstream = torch.cuda.Stream(dev)
    hctx = P.Context(ctx.device, hstream)
    keys = [torch.empty(x[6], dtype=torch.int64, device=dev) for x in inputs]
    g0s = [x[5] for x in inputs]

    def enqueue(arenas, ready_in=None):
        """Hash every interval (after its copy when ready_in is given), then the trace;
        arenas[i] = (tokens, offsets, prefix lengths, suffix lengths) of interval i."""
        pipe.reset()
        start = torch.cuda.Event()
        start.record(stream)
        hstream.wait_event(start)
        hashed = []
        for i, (tok, off, plen, _) in enumerate(arenas):
            if ready_in is not None:
                hstream.wait_event(ready_in[i])
            P.hash_prefixes(hctx, tok, off, plen, 0, out=keys[i])
            e = torch.cuda.Event()
            e.record(hstream)
            hashed.append(e)
        pipe.run(keys, [a[2] for a in arenas], [a[3] for a in arenas], g0s, ready=hashed)
        stream.wait_event(hashed[-1])

    resident = [(x[1], x[2], x[3], x[4]) for x in inputs]
    for _ in range(max(args.warmup, 1 if args.graph else 0)):  # a graph captures warm buffers only
        enqueue(resident)
    pipe.sync()
    hctx.sync()
    prof = pipe.contexts + [hctx]
    # optional CUDA graph of the whole step (every interval's hash, plans, routes and
    # replay): the host then enqueues one graph per step instead of every launch
    graph, graph_launches = None, 0
    if args.graph:
        pipe.quiesce()
        lc0 = pipe.launches + hctx.launches
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            enqueue(resident)
        graph_launches = pipe.launches + hctx.launches - lc0
        graph.replay()
        torch.cuda.synchronize()
    else:
        for c in prof:
            c.profile_enable(16 * cfg.n_intervals * max(args.steps, 1) + 64)
    clocks = ClockSampler(dev.index or 0, args.clocks_out)
    clocks.start()
    time.sleep(0.3)
    barrier()
    torch.cuda.synchronize()
    l0 = pipe.launches + hctx.launches
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        if graph is not None:
            graph.replay()
        else:
            enqueue(resident)
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    n_launch = graph_launches * args.steps if graph is not None else pipe.launches + hctx.launches - l0
    clk = clocks.stop()
    steps_profiled = args.steps
    if graph is not None:  # kernel times from one ordinary step after the timed region
        pipe.quiesce()
        for c in prof:
            c.profile_enable(16 * cfg.n_intervals + 64)
        enqueue(resident)
        steps_profiled = 1
    pipe.sync()
    kern = {}
    for tag in ("hash", "plan", "route_cand", "route_resolve", "partition", "replay"):
        n_, ms_ = 0, 0.0
        for c in prof:
            a, b = c.profile_read(tag)
            n_, ms_ = n_ + a, ms_ + b
        kern[tag] = {"launches": n_, "avg_ms": ms_ / n_ if n_ else None, "ms_per_step": ms_ / steps_profiled}
    for c in prof:
        c.profile_enable(0)
    ms = ev0.elapsed_time(ev1) / args.steps
    ms_max = max_over_ranks(ms, world, dev)
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    peak_src = "measured" if "hbm_gbs" in peaks else "fallback"
    reps, ncaps = len(cfg.replicas), len(cfg.caps)
    hb = float(np.mean(hash_bytes))
    hash_ms = kern["hash"]["avg_ms"]
    hash_rf = {"kernel": "k_hash_prefixes", "bound": "hbm", "achieved": hb / (hash_ms / 1e3) / 1e9,
               "peak": hbm_peak, "peak_source": peak_src, "unit": "GB/s",
               "frac": hb / (hash_ms / 1e3) / 1e9 / hbm_peak, "traffic": hash_traffic(hb),
               "algorithmic_bytes_per_launch_mean": hb, "avg_launch_ms": hash_ms,
               "launches_timed": kern["hash"]["launches"]}
    req_per_launch = n_step * steps_profiled / max(kern["replay"]["launches"], 1)
    a9_bytes = 20.0 * reps * ncaps * req_per_launch
    lru_ms = kern["replay"]["avg_ms"]
    lru_rf = {"kernel": "k_lru_stamp (a9 LRU replay)" if not cfg.lru_tokens else "k_lru_tokens (a9 byte-aware replay)",
              "bound": "hbm", "achieved": a9_bytes / (lru_ms / 1e3) / 1e9, "peak": hbm_peak,
              "peak_source": peak_src, "unit": "GB/s", "frac": a9_bytes / (lru_ms / 1e3) / 1e9 / hbm_peak,
              "traffic": lru_traffic(a9_bytes, reps * req_per_launch) if not cfg.lru_tokens else None,
              "algorithmic_bytes_per_launch_mean": a9_bytes, "avg_launch_ms": lru_ms,
              "requests_per_launch": req_per_launch, "launches_timed": kern["replay"]["launches"],
              "note": "20 B per (request, replica, capacity), the algorithmic bytes of the replay step"}
    # the roofline object names the kernel with the larger share of the step
    dom_lru = kern["replay"]["ms_per_step"] >= kern["hash"]["ms_per_step"]
    rr_bytes = 8 + 2 * reps + 6 * reps + 20 * reps * ncaps
    line = {
        "metric": METRIC, "value": job_throughput(n_step, world, ms_max), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": dict(workload_config(cfg, args.batch, args.fresh_plans),
                       schedule=(f"hashing on its own stream, one event per interval; {args.depth} intervals in "
                                 f"flight: plans on {args.plan_streams} streams, routes on {args.route_streams} "
                                 f"streams, the replay in interval order, {args.replay_group} intervals per call"
                                 + ("; the step captured once as a CUDA graph and replayed" if graph is not None
                                    else ""))),
        "roofline": lru_rf if dom_lru else hash_rf,
        ("hash_roofline" if dom_lru else "replay_roofline"): hash_rf if dom_lru else lru_rf,
        "kernels_ms_per_launch": kern,
        "plan_build_ms": {"mean_in_step": kern["plan"]["avg_ms"],
                          "isolated": isolated_plan_ms(pipe, keys)},
        "route_replay": {"algorithmic_bytes_per_request": rr_bytes,
                         "achieved_GBps": rr_bytes * n_step / (ms_max / 1e3) / 1e9,
                         "hbm_frac": rr_bytes * n_step / (ms_max / 1e3) / 1e9 / hbm_peak,
                         "note": "algorithmic route + replay bytes over the whole step (hashing and plans included "
                                 "in the time)"},
        "gpu_launches": int(n_launch), "clocks": clk,
    }
    if not args.no_e2e:
        line["e2e"] = e2e_resident(args, pipe, enqueue, inputs, dev, stream, n_step, world)
    if not args.no_cpu_baseline and world == 1:
        sample = oracle_interval_sample(trace)
        nproc = os.cpu_count() or 1
        t1 = oracle_interval_step(trace, sample, 1, args.batch)
        tn = oracle_interval_step(trace, sample, nproc, args.batch)
        line["cpu_baseline"] = {"value": sample["n"] / tn, "unit": UNIT, "cores": nproc, "kind": "oracle",
                                "sample": f"interval 0 of {cfg.n_intervals} ({sample['n']} requests, all "
                                          f"{len(cfg.replicas)} replicas), hash+plan+route+replay, C oracle on "
                                          f"{nproc} host threads over request ranges, plan variants and replicas",
                                "single_thread": {"value": sample["n"] / t1, "unit": UNIT, "cores": 1},
                                "nproc": nproc}
    if rank == 0:
        print(json.dumps(line), flush=True)
    pipe.close()
    hctx.close()
    if world > 1:
        dist.destroy_process_group()


def e2e_resident(args, pipe, enqueue, inputs, dev, stream, n_step, world):
    """End to end through the public API: every step copies each interval's token arena,
    offsets and lengths from pinned host memory (a copy stream, one event per interval, so
    hashing of interval t starts once its inputs have landed), runs the trace and reads
    the counters back."""
    import torch
    host, dbuf = [], []
    for (t, tok, off, plen, slen, g0, n) in inputs:
        h = []
        for x in (tok, off, plen, slen):
            p = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
            p.copy_(x)
            h.append(p)
        host.append(h)
        dbuf.append([torch.empty_like(x, device=dev) for x in h])
    h2d = sum(x.numel() * x.element_size() for h in host for x in h)
    copy_stream = torch.cuda.Stream(dev)
    out = torch.empty(pipe.ctr.shape, dtype=torch.int64, pin_memory=True)
    d2h = out.numel() * out.element_size()

    def step():
        start = torch.cuda.Event()
        start.record(stream)
        copy_stream.wait_event(start)
        ready = []
        with torch.cuda.stream(copy_stream):
            for h, d in zip(host, dbuf):
                for a, b in zip(h, d):
                    b.copy_(a, non_blocking=True)
                e = torch.cuda.Event()
                e.record(copy_stream)
                ready.append(e)
        enqueue([(d[0], d[1], d[2], d[3]) for d in dbuf], ready_in=ready)
        out.copy_(pipe.ctr, non_blocking=True)

    for _ in range(2):
        step()
    torch.cuda.synchronize()
    each = []
    for _ in range(args.e2e_steps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step()
        e1.record(stream)
        e1.synchronize()
        each.append(e0.elapsed_time(e1))
    ms = max_over_ranks(float(np.median(each)), world, dev)
    return {"value": job_throughput(n_step, world, ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "ms_per_step_each": [round(x, 2) for x in each],
            "note": "token arenas, offsets, prefix and suffix lengths of every interval copied from pinned host "
                    "memory on a copy stream each step (hashing of an interval waits for its copy), counters read "
                    "back; median of the timed steps"}


def e2e(args, ctx, pipe, inputs, dev, stream, n_step, world):
    """Same step through the public API, inputs copied from pinned host memory every step
    (copy stream overlapped with compute, double-buffered), counters read back."""
    import torch
    host = []
    h2d = 0
    for (t, tok, off, plen, slen, g0, n) in inputs:
        h = []
        for x in (tok, off, plen, slen):
            p = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
            p.copy_(x)
            h.append(p)
        h = tuple(h)
        host.append((t, h, g0, n))
        h2d += sum(x.numel() * x.element_size() for x in h)
    max_tok = max(x[1][0].numel() for x in host)
    NB = 4  # input buffers: the replay, their last reader, runs intervals behind the copies
    max_n = max(x[3] for x in host)
    bufs = [(torch.empty(max_tok, dtype=torch.int32, device=dev), torch.empty(max_n, dtype=torch.int64, device=dev),
             torch.empty(max_n, dtype=torch.int32, device=dev), torch.empty(max_n, dtype=torch.int32, device=dev))
            for _ in range(NB)]
    copy_stream = torch.cuda.Stream(dev)
    done = [torch.cuda.Event() for _ in range(NB)]     # compute finished with buffer
    ready = [torch.cuda.Event() for _ in range(NB)]    # copy into buffer finished
    out = torch.empty(pipe.ctr.shape, dtype=torch.int64, pin_memory=True)
    d2h = out.numel() * out.element_size()

    copy_marks = []

    def step(mark=False):
        pipe.reset()
        for i, (t, h, g0, n) in enumerate(host):
            b = i % NB
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(done[b])
                if mark:
                    c0 = torch.cuda.Event(enable_timing=True)
                    c0.record(copy_stream)
                dtok, doff, dpl, dsl = bufs[b]
                ntok = h[0].numel()
                dtok[:ntok].copy_(h[0], non_blocking=True)
                doff[:n].copy_(h[1], non_blocking=True)
                dpl[:n].copy_(h[2], non_blocking=True)
                dsl[:n].copy_(h[3], non_blocking=True)
                ready[b].record(copy_stream)
                if mark:
                    c1 = torch.cuda.Event(enable_timing=True)
                    c1.record(copy_stream)
                    copy_marks.append((c0, c1))
            stream.wait_event(ready[b])
            dtok, doff, dpl, dsl = bufs[b]
            pipe.interval(t, dtok[:h[0].numel()], doff[:n], dpl[:n], dsl[:n], g0, plan_next=i + 1 < len(host),
                          inputs_ready=ready[b])
            done[b] = pipe.inputs_free   # after this interval's replay, the last reader of its inputs
        pipe.finish()
        out.copy_(pipe.ctr, non_blocking=True)

    for _ in range(2):
        step()
    torch.cuda.synchronize()
    # every step timed on its own: copies over the host link are now and then slowed by other
    # traffic on the shared host, so the median step is reported and every step listed
    each = []
    for k in range(args.e2e_steps):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        step(mark=k == args.e2e_steps - 1)
        e1.record(stream)  # after the counters' read-back on this stream
        e1.synchronize()
        each.append(e0.elapsed_time(e1))
    ms = max_over_ranks(float(np.median(each)), world, dev)
    copy_ms = float(sum(a.elapsed_time(b) for a, b in copy_marks))
    return {"value": job_throughput(n_step, world, ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "ms_per_step_each": [round(x, 2) for x in each],
            "mean_ms_per_step": float(np.mean(each)),
            "h2d_copy_ms_per_step": copy_ms, "h2d_GBps_while_copying": h2d / (copy_ms / 1e3) / 1e9,
            "note": "pinned host -> HBM copies on a second stream overlapped with compute (four buffers); "
                    "median of the timed steps (each step timed alone; the host-link copies of some steps "
                    "are slowed by other traffic on the shared host); copy times from events on the copy "
                    "stream in the last step"}


if __name__ == "__main__":
    main()
