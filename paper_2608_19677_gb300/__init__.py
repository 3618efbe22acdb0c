"""GB300 (sm_103a) hot path of planned prefix-affinity routing (CacheRoute, arXiv 2608.19677).

Thin ctypes binding over the C ABI declared in ``include/cacheroute.h``: every
function below only marshals torch CUDA tensors into device pointers and calls
the library of the same name; every step of the path runs in the library's
CUDA kernels.  There is no CPU fallback: importing works without a GPU, but
creating a ``Context`` requires the compiled library and a CUDA device, and
fails loudly otherwise.

  hash_prefixes   request prefix spans -> routing keys          (cr_hash_prefixes)
  build_plans     one interval's keys -> plans (Eq. 1, Alg. 1)  (cr_build_plans)
  route_batch     keys -> destination per (request, replica)    (cr_route_batch)
  Ring            ring of the bounded-load policy               (cr_ring_create)
  plan_diff       churn between two plans                       (cr_plan_diff)
  shadow_replay   routed requests -> LRU hit / load counters    (cr_shadow_replay)
"""
from __future__ import annotations

import ctypes as C
import os
from typing import List, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# CR_DEBUG_LIB=1 loads the bounds-checking build (buildlib.build(debug=True)) instead
LIB_PATH = os.path.join(_HERE, "libcacheroute_debug.so" if os.environ.get("CR_DEBUG_LIB") == "1"
                        else "libcacheroute.so")

CR_OK, CR_EINVAL, CR_ENOMEM, CR_ECUDA, CR_ETIMEOUT, CR_EOVERFLOW = range(6)
STATUS_NAMES = {0: "CR_OK", 1: "CR_EINVAL", 2: "CR_ENOMEM", 3: "CR_ECUDA", 4: "CR_ETIMEOUT",
                5: "CR_EOVERFLOW"}
POLICY = {"CR": 0, "CR_NOLPT": 1, "CR_NOREPL": 2, "P2C": 3, "RR": 4, "HASH": 5, "CHWBL": 6}
VARIANT = {"LPT": 0, "RANDOM": 1, "NOREPL": 2, "SLOTCAP": 3}
MAX_R, MAX_CAP, MAX_CAPS, MAX_REPLICAS, CTR_FIELDS, MAX_VNODES = 8192, 1024, 8, 256, 5, 1024

# every symbol the header declares (checked by the CPU test suite)
EXPORTS = ("cr_create", "cr_destroy", "cr_set_stream", "cr_sync", "cr_last_error", "cr_launch_count",
           "cr_hash_prefixes", "cr_plan_create", "cr_plan_destroy", "cr_build_plans", "cr_build_plan",
           "cr_plan_get_info", "cr_plan_export", "cr_route_batch", "cr_replay_create", "cr_replay_reset",
           "cr_replay_destroy", "cr_shadow_replay", "cr_replay_export_state", "cr_key_histogram_noalloc",
           "cr_ring_create", "cr_ring_destroy", "cr_ring_export", "cr_plan_diff",
           "cr_replay_create_tokens", "cr_set_resolve_stream", "cr_partition_create", "cr_partition_destroy",
           "cr_profile_enable", "cr_profile_read", "cr_plan_import", "cr_replay_import_state",
           "cr_replay_input_create", "cr_replay_input_destroy", "cr_replay_partition", "cr_replay_simulate")
PROF = {"hash": 0, "plan": 1, "route_cand": 2, "route_resolve": 3, "partition": 4, "replay": 5}
CR_NOALLOC_MAX_KEYS = 65536


class CacheRouteError(RuntimeError):
    def __init__(self, code: int, where: str, msg: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


class PlanParams(C.Structure):
    _fields_ = [("R", C.c_uint32), ("W", C.c_uint32), ("qcap_num", C.c_uint64),
                ("qcap_den", C.c_uint64), ("variant", C.c_uint32), ("reserved", C.c_uint32),
                ("seed", C.c_uint64), ("epoch", C.c_uint64), ("d_init_load", C.c_void_p)]


class PlanInfo(C.Structure):
    _fields_ = [("n", C.c_uint64), ("U", C.c_uint64), ("n_adm", C.c_uint64), ("sum_k", C.c_uint64),
                ("cold", C.c_uint64), ("max_k", C.c_uint64), ("R", C.c_uint32), ("W", C.c_uint32)]


class PlanDiff(C.Structure):
    _fields_ = [(f, C.c_uint64) for f in ("keys_a", "keys_b", "keys_common", "pairs_a", "pairs_b",
                                          "pairs_common", "adm_k_changed", "adm_set_changed", "hist_keys",
                                          "hist_kb_changed")]


class Replica(C.Structure):
    _fields_ = [("policy", C.c_uint32), ("reserved", C.c_uint32), ("seed", C.c_uint64), ("ring", C.c_void_p)]


_lib = None


def build(force: bool = False) -> str:
    """Compile the CUDA library in-tree (nvcc, sm_103a)."""
    from . import buildlib
    return buildlib.build(force=force)


def lib() -> C.CDLL:
    """The loaded CUDA library; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build the CUDA library first "
                          f"(python -c 'import __graft_entry__ as g; g.build()')")
    L = C.CDLL(LIB_PATH)
    vp, u64, u32, i32 = C.c_void_p, C.c_uint64, C.c_uint32, C.c_int
    sig = {
        "cr_create": ([C.POINTER(vp), i32, vp], i32),
        "cr_destroy": ([vp], i32),
        "cr_set_stream": ([vp, vp], i32),
        "cr_sync": ([vp], i32),
        "cr_last_error": ([vp], C.c_char_p),
        "cr_launch_count": ([vp], u64),
        "cr_hash_prefixes": ([vp, vp, vp, vp, u64, u64, vp], i32),
        "cr_plan_create": ([vp, C.POINTER(vp)], i32),
        "cr_plan_destroy": ([vp, vp], i32),
        "cr_build_plans": ([vp, vp, u64, C.POINTER(PlanParams), u32, C.POINTER(vp)], i32),
        "cr_build_plan": ([vp, vp, u64, C.POINTER(PlanParams), vp], i32),
        "cr_plan_get_info": ([vp, vp, C.POINTER(PlanInfo)], i32),
        "cr_plan_export": ([vp, vp] + [vp] * 9, i32),
        "cr_route_batch": ([vp, C.POINTER(vp), C.POINTER(Replica), u32, u32, vp, u64, u64, u32, vp, vp], i32),
        "cr_replay_create": ([vp, u32, u32, C.POINTER(C.c_uint32), u32, C.POINTER(vp)], i32),
        "cr_replay_create_tokens": ([vp, u32, u32, C.POINTER(C.c_uint32), u32, C.POINTER(vp)], i32),
        "cr_replay_reset": ([vp, vp], i32),
        "cr_replay_destroy": ([vp, vp], i32),
        "cr_shadow_replay": ([vp, vp, vp, vp, vp, vp, u64, vp], i32),
        "cr_replay_export_state": ([vp, vp, u32, u32, vp, C.POINTER(C.c_uint32)], i32),
        "cr_key_histogram_noalloc": ([vp, u64, vp, vp, vp, vp], i32),
        "cr_ring_create": ([vp, u32, u32, u64, C.POINTER(vp)], i32),
        "cr_ring_destroy": ([vp, vp], i32),
        "cr_ring_export": ([vp, vp, vp, vp], i32),
        "cr_plan_diff": ([vp, vp, vp, C.POINTER(PlanDiff)], i32),
        "cr_set_resolve_stream": ([vp, vp], i32),
        "cr_partition_create": ([i32, u32, C.POINTER(vp), C.POINTER(vp), C.POINTER(vp)], i32),
        "cr_partition_destroy": ([vp], i32),
        "cr_plan_import": ([vp, vp, u32, u32, u64, vp, vp, vp, vp, vp, vp], i32),
        "cr_replay_import_state": ([vp, vp, u32, u32, vp, u32], i32),
        "cr_replay_input_create": ([vp, C.POINTER(vp)], i32),
        "cr_replay_input_destroy": ([vp, vp], i32),
        "cr_replay_partition": ([vp, vp, vp, vp, vp, vp, u64, vp], i32),
        "cr_replay_simulate": ([vp, vp, vp, vp], i32),
        "cr_profile_enable": ([vp, u32], i32),
        "cr_profile_read": ([vp, u32, C.POINTER(C.c_uint64), C.POINTER(C.c_double)], i32),
    }
    for name, (args, res) in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res
    _lib = L
    return L


def _ptr(t) -> int:
    return 0 if t is None else int(t.data_ptr())


def _np_ptr(a: np.ndarray):
    return a.ctypes.data_as(C.c_void_p)


class Context:
    """A library context bound to one CUDA device and stream (torch's current stream by default)."""

    def __init__(self, device: int = 0, stream=None):
        import torch
        self.device = device
        self._stream_obj = stream if stream is not None else torch.cuda.current_stream(device)
        h = C.c_void_p()
        st = lib().cr_create(C.byref(h), device, C.c_void_p(self._stream_obj.cuda_stream))
        if st != CR_OK:
            raise CacheRouteError(st, "cr_create", lib().cr_last_error(None).decode())
        self._h = h

    @property
    def handle(self):
        return self._h

    def check(self, st: int, where: str):
        if st != CR_OK:
            raise CacheRouteError(st, where, lib().cr_last_error(self._h).decode())

    def sync(self):
        self.check(lib().cr_sync(self._h), "cr_sync")

    def set_stream(self, stream):
        self._stream_obj = stream
        self.check(lib().cr_set_stream(self._h, C.c_void_p(stream.cuda_stream)), "cr_set_stream")

    @property
    def launches(self) -> int:
        return int(lib().cr_launch_count(self._h))

    def profile_enable(self, max_launches: int):
        """Time the library's main kernels per launch with CUDA events (0: off); forgets earlier launches."""
        self.check(lib().cr_profile_enable(self._h, max_launches), "cr_profile_enable")

    def profile_read(self, tag: str):
        """(timed launches, summed milliseconds) of one kind of launch (blocking)."""
        n, ms = C.c_uint64(), C.c_double()
        self.check(lib().cr_profile_read(self._h, PROF[tag], C.byref(n), C.byref(ms)), "cr_profile_read")
        return int(n.value), float(ms.value)

    def close(self):
        if getattr(self, "_h", None):
            lib().cr_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _need_cuda(name, t, dtype=None):
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must have dtype {dtype}, got {t.dtype}")


def hash_prefixes(ctx: Context, tokens, off, plen, salt: int = 0, out=None):
    """Routing key per request (uint64 values in an int64 tensor)."""
    import torch
    n = int(off.shape[0])
    _need_cuda("tokens", tokens, torch.int32)
    _need_cuda("off", off, torch.int64)
    _need_cuda("plen", plen, torch.int32)
    if out is None:
        out = torch.empty(n, dtype=torch.int64, device=off.device)
    ctx.check(lib().cr_hash_prefixes(ctx.handle, _ptr(tokens), _ptr(off), _ptr(plen), n,
                                     salt & ((1 << 64) - 1), _ptr(out)), "cr_hash_prefixes")
    return out


class Plan:
    """A library-owned plan (device resident)."""

    def __init__(self, ctx: Context):
        self.ctx = ctx
        h = C.c_void_p()
        ctx.check(lib().cr_plan_create(ctx.handle, C.byref(h)), "cr_plan_create")
        self._h = h

    @property
    def handle(self):
        return self._h

    def info(self) -> PlanInfo:
        inf = PlanInfo()
        self.ctx.check(lib().cr_plan_get_info(self.ctx.handle, self._h, C.byref(inf)), "cr_plan_get_info")
        return inf

    def export(self) -> dict:
        inf = self.info()
        U, na, sk, R = int(inf.U), int(inf.n_adm), int(inf.sum_k), int(inf.R)
        a = dict(ukey=np.zeros(max(U, 1), np.uint64), ucnt=np.zeros(max(U, 1), np.uint64),
                 adm_key=np.zeros(max(na, 1), np.uint64), adm_cnt=np.zeros(max(na, 1), np.uint64),
                 adm_k=np.zeros(max(na, 1), np.uint32), koff=np.zeros(na + 1, np.uint32),
                 members=np.zeros(max(sk, 1), np.uint16), jobs=np.zeros(max(sk, 1), np.uint64),
                 load=np.zeros(R, np.uint64))
        self.ctx.check(lib().cr_plan_export(self.ctx.handle, self._h, *[_np_ptr(a[k]) for k in
                                                                        ("ukey", "ucnt", "adm_key", "adm_cnt",
                                                                         "adm_k", "koff", "members", "jobs",
                                                                         "load")]), "cr_plan_export")
        out = dict(U=U, n_adm=na, sum_k=sk, cold=int(inf.cold), max_k=int(inf.max_k), R=R, W=int(inf.W))
        out.update(ukey=a["ukey"][:U], ucnt=a["ucnt"][:U], adm_key=a["adm_key"][:na], adm_cnt=a["adm_cnt"][:na],
                   adm_k=a["adm_k"][:na], koff=a["koff"], members=a["members"][:sk], jobs=a["jobs"][:sk],
                   load=a["load"])
        return out

    def load(self, R: int, W: int, adm_key, adm_cnt, adm_k, members, jobs=None, load=None):
        """Install a plan given as host arrays in admission order (cr_plan_import)."""
        ak = np.ascontiguousarray(adm_key, np.uint64)
        ac = np.ascontiguousarray(adm_cnt, np.uint64)
        kk = np.ascontiguousarray(adm_k, np.uint32)
        mm = np.ascontiguousarray(members, np.uint16)
        jb = None if jobs is None else np.ascontiguousarray(jobs, np.uint64)
        ld = None if load is None else np.ascontiguousarray(load, np.uint64)
        self.ctx.check(lib().cr_plan_import(self.ctx.handle, self._h, R, W, ak.size, _np_ptr(ak), _np_ptr(ac),
                                            _np_ptr(kk), _np_ptr(mm), None if jb is None else _np_ptr(jb),
                                            None if ld is None else _np_ptr(ld)), "cr_plan_import")
        return self

    def close(self):
        if getattr(self, "_h", None):
            lib().cr_plan_destroy(self.ctx.handle, self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def plan_params(R: int, W: int, qcap_num: int, qcap_den: int, variant="LPT", seed: int = 0, epoch: int = 0,
                init_load=None) -> PlanParams:
    v = VARIANT[variant] if isinstance(variant, str) else int(variant)
    p = PlanParams(R, W, qcap_num, qcap_den, v, 0, seed & ((1 << 64) - 1), epoch, _ptr(init_load))
    p._init_load = init_load  # the device vector must outlive the parameters that point at it
    return p


def build_plans(ctx: Context, keys, params: Sequence[PlanParams], plans: Sequence[Plan]):
    import torch
    n = int(keys.shape[0])
    _need_cuda("keys", keys, torch.int64)
    arr = (PlanParams * len(params))(*params)
    hs = (C.c_void_p * len(plans))(*[p.handle for p in plans])
    ctx.check(lib().cr_build_plans(ctx.handle, _ptr(keys), n, arr, len(params), hs), "cr_build_plans")
    return plans


def build_plan(ctx: Context, keys, params: PlanParams, plan: Optional[Plan] = None) -> Plan:
    plan = plan or Plan(ctx)
    build_plans(ctx, keys, [params], [plan])
    return plan


def set_resolve_stream(ctx: Context, stream) -> None:
    """Route with the load-dependent resolution on ``stream`` (a torch stream; None: the context's)."""
    ctx.check(lib().cr_set_resolve_stream(ctx.handle, C.c_void_p(stream.cuda_stream) if stream is not None
                                          else None), "cr_set_resolve_stream")


class Partition:
    """Two streams whose kernels run on disjoint SM sets (green contexts): ``big`` and ``small``
    (torch external streams; ``small`` has ``small_sms`` SMs)."""

    def __init__(self, device: int, small_sms: int):
        import torch
        h, b, sm = C.c_void_p(), C.c_void_p(), C.c_void_p()
        st = lib().cr_partition_create(device, small_sms, C.byref(h), C.byref(b), C.byref(sm))
        if st != CR_OK:
            raise CacheRouteError(st, "cr_partition_create", lib().cr_last_error(None).decode())
        self._h = h
        dev = torch.device("cuda", device)
        self.big = torch.cuda.ExternalStream(b.value, device=dev)
        self.small = torch.cuda.ExternalStream(sm.value, device=dev)

    def close(self):
        if getattr(self, "_h", None):
            lib().cr_partition_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def plan_diff(ctx: Context, a: Plan, b: Plan) -> dict:
    """Counts of how plan b differs from plan a (blocking); see ``churn``."""
    out = PlanDiff()
    ctx.check(lib().cr_plan_diff(ctx.handle, a.handle, b.handle, C.byref(out)), "cr_plan_diff")
    return {f: int(getattr(out, f)) for f, _ in PlanDiff._fields_}


def churn(diff: dict):
    """(cache churn, count churn) as floats: 1 - Jaccard of the assignment sets, and the share of
    the keys of either histogram whose Eq. 1 k_b changed."""
    up = diff["pairs_a"] + diff["pairs_b"] - diff["pairs_common"]
    return (1.0 - diff["pairs_common"] / up if up else 0.0,
            diff["hist_kb_changed"] / diff["hist_keys"] if diff["hist_keys"] else 0.0)


class Ring:
    """Consistent-hashing ring of the bounded-load policy (R destinations x vnodes points), on the device."""

    def __init__(self, ctx: Context, R: int, vnodes: int, seed: int):
        self.ctx, self.R, self.vnodes, self.seed = ctx, R, vnodes, seed & ((1 << 64) - 1)
        h = C.c_void_p()
        ctx.check(lib().cr_ring_create(ctx.handle, R, vnodes, self.seed, C.byref(h)), "cr_ring_create")
        self._h = h

    @property
    def handle(self):
        return self._h

    def export(self):
        """(point uint64 [R*vnodes] ascending, owner uint16 [R*vnodes]) on the host."""
        M = self.R * self.vnodes
        pt = np.zeros(M, np.uint64)
        ow = np.zeros(M, np.uint16)
        self.ctx.check(lib().cr_ring_export(self.ctx.handle, self._h, _np_ptr(pt), _np_ptr(ow)), "cr_ring_export")
        return pt, ow

    def close(self):
        if getattr(self, "_h", None):
            lib().cr_ring_destroy(self.ctx.handle, self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def route_batch(ctx: Context, plans: Sequence[Optional[Plan]], policies: Sequence, seeds: Sequence[int],
                R: int, keys, first_req_index: int, batch_B: int, load, dest=None,
                rings: Optional[Sequence[Optional[Ring]]] = None):
    """Destinations (uint16 values in an int16 tensor [n_rep, n]); ``load`` [n_rep, R] is updated in place.

    ``rings[i]`` is the ring of replica i when its policy is CHWBL."""
    import torch
    n_rep = len(policies)
    n = int(keys.shape[0])
    _need_cuda("keys", keys, torch.int64)
    _need_cuda("load", load, torch.int64)
    if dest is None:
        dest = torch.empty((n_rep, n), dtype=torch.int16, device=keys.device)
    _need_cuda("dest", dest, torch.int16)
    rg = list(rings) if rings is not None else [None] * n_rep
    reps = (Replica * n_rep)(*[Replica(POLICY[p] if isinstance(p, str) else int(p), 0,
                                       int(s) & ((1 << 64) - 1), (g.handle.value if g is not None else None))
                               for p, s, g in zip(policies, seeds, rg)])
    hs = (C.c_void_p * n_rep)(*[(p.handle if p is not None else None) for p in plans])
    ctx.check(lib().cr_route_batch(ctx.handle, hs, reps, n_rep, R, _ptr(keys), n, first_req_index, batch_B,
                                   _ptr(load), _ptr(dest)), "cr_route_batch")
    return dest


class Replay:
    """Library-owned LRU state for n_rep x R destinations x len(caps) capacities.

    ``tokens``: capacities count prefix tokens (byte-aware variant, cr_replay_create_tokens)."""

    def __init__(self, ctx: Context, n_rep: int, R: int, caps: Sequence[int], tokens: bool = False):
        self.ctx, self.n_rep, self.R, self.caps, self.tokens = ctx, n_rep, R, list(caps), tokens
        cp = (C.c_uint32 * len(caps))(*caps)
        h = C.c_void_p()
        name = "cr_replay_create_tokens" if tokens else "cr_replay_create"
        ctx.check(getattr(lib(), name)(ctx.handle, n_rep, R, cp, len(caps), C.byref(h)), name)
        self._h = h

    @property
    def handle(self):
        return self._h

    def reset(self):
        self.ctx.check(lib().cr_replay_reset(self.ctx.handle, self._h), "cr_replay_reset")

    def set_state(self, rep: int, r: int, keys):
        """Resident keys of one simulator, most recent first (cr_replay_import_state)."""
        k = np.ascontiguousarray(keys, np.uint64)
        self.ctx.check(lib().cr_replay_import_state(self.ctx.handle, self._h, rep, r,
                                                    _np_ptr(k) if k.size else None, k.size), "cr_replay_import_state")

    def state(self, rep: int, r: int) -> np.ndarray:
        out = np.zeros(MAX_CAP, np.uint64)
        fill = C.c_uint32()
        self.ctx.check(lib().cr_replay_export_state(self.ctx.handle, self._h, rep, r, _np_ptr(out),
                                                    C.byref(fill)), "cr_replay_export_state")
        return out[:fill.value].copy()

    def close(self):
        if getattr(self, "_h", None):
            lib().cr_replay_destroy(self.ctx.handle, self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class ReplayInput:
    """A partitioned batch of routed requests (cr_replay_partition), read by replay_simulate."""

    def __init__(self, ctx: Context):
        self.ctx = ctx
        h = C.c_void_p()
        ctx.check(lib().cr_replay_input_create(ctx.handle, C.byref(h)), "cr_replay_input_create")
        self._h = h

    @property
    def handle(self):
        return self._h

    def close(self):
        if getattr(self, "_h", None):
            lib().cr_replay_input_destroy(self.ctx.handle, self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def replay_partition(ctx: Context, replay: Replay, keys, plen, slen, dest, inp: ReplayInput):
    """Partition routed requests for `replay` into `inp` (a8 alone), on ctx's stream."""
    import torch
    n = int(keys.shape[0])
    _need_cuda("keys", keys, torch.int64)
    _need_cuda("plen", plen, torch.int32)
    _need_cuda("slen", slen, torch.int32)
    _need_cuda("dest", dest, torch.int16)
    ctx.check(lib().cr_replay_partition(ctx.handle, replay.handle, _ptr(keys), _ptr(plen), _ptr(slen), _ptr(dest),
                                        n, inp.handle), "cr_replay_partition")
    return inp


def replay_simulate(ctx: Context, replay: Replay, inp: ReplayInput, ctr):
    """Run the simulators over a partitioned input (a9 alone), accumulating into ``ctr``."""
    import torch
    _need_cuda("ctr", ctr, torch.int64)
    ctx.check(lib().cr_replay_simulate(ctx.handle, replay.handle, inp.handle, _ptr(ctr)), "cr_replay_simulate")
    return ctr


def shadow_replay(ctx: Context, replay: Replay, keys, plen, slen, dest, ctr):
    """Accumulate counters into ``ctr`` (int64 [n_rep, n_caps, R, 5])."""
    import torch
    n = int(keys.shape[0])
    _need_cuda("keys", keys, torch.int64)
    _need_cuda("plen", plen, torch.int32)
    _need_cuda("slen", slen, torch.int32)
    _need_cuda("dest", dest, torch.int16)
    _need_cuda("ctr", ctr, torch.int64)
    ctx.check(lib().cr_shadow_replay(ctx.handle, replay.handle, _ptr(keys), _ptr(plen), _ptr(slen), _ptr(dest),
                                     n, _ptr(ctr)), "cr_shadow_replay")
    return ctr
