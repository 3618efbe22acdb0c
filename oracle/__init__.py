"""CPU oracle for the planned prefix-affinity routing hot path (ctypes wrapper).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package; the library under
``paper_2608_19677_gb300`` never does.  The C source ``cr_oracle.c`` is a plain,
slow, single-threaded restatement of the paper's Eq. 1 and Algorithm 1, of its
dispatch rule (Fig. 1, sec. 3.1) and of the whole-prefix LRU replay this
library adopts for the shadow-replay gate (sec. 3.2, 5.3).  It shares no code with
the CUDA path.

Parity status per function (what pins it; see tests/test_oracle_*.py):
  fmix64 / Philox4x64-10 .. published SplitMix64 outputs; numpy's Philox.
  hash_prefixes ........... published SplitMix64 outputs on all-zero spans,
                            the additive-by-position identity, sensitivity.
  histogram ............... collections.Counter; conservation.
  build_plan .............. hand-worked example (tests/golden), brute-force
                            admission, Graham's LPT bound by brute force,
                            job conservation, Eq. 1 by exact fractions,
                            "every k_b = 1 when max lambda < q_cap".
  route ................... conservation, round-robin balance, hash
                            stickiness and jump-hash monotonicity, P2C by a
                            hand-stepped sequence, admitted keys land in T(b).
  shadow_replay ........... hand trace, infinite-capacity closed form,
                            capacity-1 rule, brute-force stack distances
                            (Mattson inclusion).
  Ring / route CHWBL ...... published SplitMix64 outputs, brute-force
                            clockwise-distance walk, exact inverse-mixer edge
                            keys, the sequential load bound, plain consistent
                            hashing when unsaturated.
  plan_diff / churn ....... hand-built plans, Jaccard of key x destination
                            incidence matrices, identity and symmetry, the
                            all-move / no-count-change case.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from typing import List, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "cr_oracle.c")
_LIB = os.path.join(_HERE, "libcr_oracle.so")

CTR_FIELDS = ("requests", "hits", "hit_tokens", "prompt_tokens", "prefill_tokens")
VARIANT = {"LPT": 0, "RANDOM": 1, "NOREPL": 2, "SLOTCAP": 3}
POLICY = {"CR": 0, "CR_NOLPT": 1, "CR_NOREPL": 2, "P2C": 3, "RR": 4, "HASH": 5, "CHWBL": 6}


def build(force: bool = False) -> str:
    """Compile the oracle with the host C compiler (plain C11, no intrinsics)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-std=gnu11", "-O2", "-fPIC", "-shared", "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        u64p, u32p, u16p, i32p = (C.POINTER(C.c_uint64), C.POINTER(C.c_uint32),
                                  C.POINTER(C.c_uint16), C.POINTER(C.c_int32))
        _lib.orc_fmix64.restype = C.c_uint64
        _lib.orc_fmix64.argtypes = [C.c_uint64]
        _lib.orc_philox4x64_10.argtypes = [u64p, u64p, u64p]
        _lib.orc_hash_one.restype = C.c_uint64
        _lib.orc_hash_one.argtypes = [i32p, C.c_uint32, C.c_uint64]
        _lib.orc_hash_prefixes.argtypes = [i32p, u64p, u32p, C.c_uint64, C.c_uint64, u64p]
        _lib.orc_histogram.restype = C.c_uint64
        _lib.orc_histogram.argtypes = [u64p, C.c_uint64, u64p, u64p]
        _lib.orc_kb.restype = C.c_uint32
        _lib.orc_kb.argtypes = [C.c_uint64, C.c_uint64, C.c_uint64, C.c_uint32]
        _lib.orc_build_plan.restype = C.c_int
        _lib.orc_build_plan.argtypes = [u64p, C.c_uint64, C.c_void_p, C.c_void_p]
        _lib.orc_jump_hash.restype = C.c_uint32
        _lib.orc_jump_hash.argtypes = [C.c_uint64, C.c_uint32]
        _lib.orc_route.restype = C.c_int
        _lib.orc_route.argtypes = [C.c_void_p, C.c_void_p, u32p, u64p, C.c_uint32, C.c_uint32, u64p,
                                   C.c_uint64, C.c_uint64, C.c_uint32, u64p, u16p]
        _lib.orc_ring_create.restype = C.c_void_p
        _lib.orc_ring_create.argtypes = [C.c_uint32, C.c_uint32, C.c_uint64]
        _lib.orc_ring_free.argtypes = [C.c_void_p]
        _lib.orc_ring_export.argtypes = [C.c_void_p, u64p, u16p]
        _lib.orc_replay_create.restype = C.c_void_p
        _lib.orc_replay_create.argtypes = [C.c_uint32, C.c_uint32, u32p, C.c_uint32]
        _lib.orc_replay_create_tokens.restype = C.c_void_p
        _lib.orc_replay_create_tokens.argtypes = [C.c_uint32, C.c_uint32, u32p, C.c_uint32]
        _lib.orc_replay_free.argtypes = [C.c_void_p]
        _lib.orc_shadow_replay.restype = C.c_int
        _lib.orc_shadow_replay.argtypes = [C.c_void_p, u64p, u32p, u32p, u16p, C.c_uint64, u64p]
        _lib.orc_replay_state.restype = C.c_uint32
        _lib.orc_replay_state.argtypes = [C.c_void_p, C.c_uint32, C.c_uint32, C.c_uint32, u64p]
    return _lib


def _p(a: np.ndarray, ct):
    return a.ctypes.data_as(C.POINTER(ct))


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# -- mixing functions ------------------------------------------------------
def fmix64(z: int) -> int:
    return int(lib().orc_fmix64(z & ((1 << 64) - 1)))


def philox4x64_10(ctr: Sequence[int], key: Sequence[int]) -> List[int]:
    c = _c(ctr, np.uint64)
    k = _c(key, np.uint64)
    o = np.zeros(4, dtype=np.uint64)
    lib().orc_philox4x64_10(_p(c, C.c_uint64), _p(k, C.c_uint64), _p(o, C.c_uint64))
    return [int(x) for x in o]


def jump_hash(k: int, R: int) -> int:
    return int(lib().orc_jump_hash(k & ((1 << 64) - 1), R))


def kb(lam: int, num: int, den: int, R: int) -> int:
    return int(lib().orc_kb(lam, num, den, R))


# -- a1 ----------------------------------------------------------------------
def hash_one(tokens, salt: int = 0) -> int:
    t = _c(tokens, np.int32)
    if t.size == 0:
        t = np.zeros(1, dtype=np.int32)
        return int(lib().orc_hash_one(_p(t, C.c_int32), 0, salt))
    return int(lib().orc_hash_one(_p(t, C.c_int32), int(np.asarray(tokens).size), salt))


def hash_prefixes(tokens, off, plen, salt: int = 0) -> np.ndarray:
    t = _c(tokens, np.int32)
    if t.size == 0:
        t = np.zeros(1, dtype=np.int32)
    o = _c(off, np.uint64)
    p = _c(plen, np.uint32)
    out = np.zeros(o.shape[0], dtype=np.uint64)
    lib().orc_hash_prefixes(_p(t, C.c_int32), _p(o, C.c_uint64), _p(p, C.c_uint32),
                            o.shape[0], salt & ((1 << 64) - 1), _p(out, C.c_uint64))
    return out


# -- a2 ----------------------------------------------------------------------
def histogram(keys):
    k = _c(keys, np.uint64)
    n = k.shape[0]
    uk = np.zeros(max(n, 1), dtype=np.uint64)
    ct = np.zeros(max(n, 1), dtype=np.uint64)
    U = lib().orc_histogram(_p(k, C.c_uint64), n, _p(uk, C.c_uint64), _p(ct, C.c_uint64))
    return uk[:U].copy(), ct[:U].copy()


# -- a3..a6 --------------------------------------------------------------------
class _Params(C.Structure):
    _fields_ = [("R", C.c_uint32), ("W", C.c_uint32), ("qcap_num", C.c_uint64),
                ("qcap_den", C.c_uint64), ("variant", C.c_uint32), ("seed", C.c_uint64),
                ("epoch", C.c_uint64), ("init_load", C.POINTER(C.c_uint64))]


class _Plan(C.Structure):
    _fields_ = [("U", C.c_uint64), ("n_adm", C.c_uint64), ("sum_k", C.c_uint64),
                ("cold", C.c_uint64),
                ("adm_key", C.POINTER(C.c_uint64)), ("adm_cnt", C.POINTER(C.c_uint64)),
                ("adm_k", C.POINTER(C.c_uint32)), ("koff", C.POINTER(C.c_uint32)),
                ("members", C.POINTER(C.c_uint16)), ("jobs", C.POINTER(C.c_uint64)),
                ("load", C.POINTER(C.c_uint64))]


class Plan:
    """A plan as plain numpy arrays (admission order)."""

    def __init__(self, R, W, U, n_adm, sum_k, cold, adm_key, adm_cnt, adm_k, koff, members,
                 jobs, load):
        self.R, self.W, self.U, self.n_adm, self.sum_k, self.cold = R, W, U, n_adm, sum_k, cold
        self.adm_key, self.adm_cnt, self.adm_k = adm_key, adm_cnt, adm_k
        self.koff, self.members, self.jobs, self.load = koff, members, jobs, load
        self._keep = None
        # set by build_plan: the interval's histogram and the plan's Eq. 1 inputs
        self.hist_key = np.zeros(0, np.uint64)
        self.hist_cnt = np.zeros(0, np.uint64)
        self.qcap = (1, 1)
        self.variant = "LPT"

    def table(self):
        """{key: [members...]} for every admitted key."""
        return {int(self.adm_key[a]): [int(m) for m in
                                        self.members[self.koff[a]:self.koff[a + 1]]]
                for a in range(self.n_adm)}

    def _struct(self):
        arrs = dict(adm_key=_c(self.adm_key, np.uint64), adm_cnt=_c(self.adm_cnt, np.uint64),
                    adm_k=_c(self.adm_k, np.uint32), koff=_c(self.koff, np.uint32),
                    members=_c(self.members, np.uint16), jobs=_c(self.jobs, np.uint64),
                    load=_c(self.load, np.uint64))
        for k, v in list(arrs.items()):
            if v.size == 0:
                arrs[k] = np.zeros(1, dtype=v.dtype)
        s = _Plan(self.U, self.n_adm, self.sum_k, self.cold,
                  _p(arrs["adm_key"], C.c_uint64), _p(arrs["adm_cnt"], C.c_uint64),
                  _p(arrs["adm_k"], C.c_uint32), _p(arrs["koff"], C.c_uint32),
                  _p(arrs["members"], C.c_uint16), _p(arrs["jobs"], C.c_uint64),
                  _p(arrs["load"], C.c_uint64))
        self._keep = arrs
        return s


def build_plan(keys, R: int, W: int, qcap_num: int, qcap_den: int, variant="LPT",
               seed: int = 0, epoch: int = 0, init_load=None) -> Plan:
    k = _c(keys, np.uint64)
    n = k.shape[0]
    C_ = R * W
    cap = max(n, 1)
    adm_key = np.zeros(cap, np.uint64)
    adm_cnt = np.zeros(cap, np.uint64)
    adm_k = np.zeros(cap, np.uint32)
    koff = np.zeros(cap + 1, np.uint32)
    members = np.zeros(max(C_, 1), np.uint16)
    jobs = np.zeros(max(C_, 1), np.uint64)
    load = np.zeros(R, np.uint64)
    il = None
    if init_load is not None:
        il = _c(init_load, np.uint64)
    prm = _Params(R, W, qcap_num, qcap_den, VARIANT[variant] if isinstance(variant, str) else variant,
                  seed, epoch, _p(il, C.c_uint64) if il is not None else None)
    pl = _Plan(0, 0, 0, 0, _p(adm_key, C.c_uint64), _p(adm_cnt, C.c_uint64),
               _p(adm_k, C.c_uint32), _p(koff, C.c_uint32), _p(members, C.c_uint16),
               _p(jobs, C.c_uint64), _p(load, C.c_uint64))
    kk = k if n else np.zeros(1, np.uint64)
    rc = lib().orc_build_plan(_p(kk, C.c_uint64), n, C.byref(prm), C.byref(pl))
    if rc != 0:
        raise ValueError(f"orc_build_plan: status {rc}")
    na, sk = int(pl.n_adm), int(pl.sum_k)
    out = Plan(R, W, int(pl.U), na, sk, int(pl.cold), adm_key[:na].copy(), adm_cnt[:na].copy(),
               adm_k[:na].copy(), koff[:na + 1].copy(), members[:sk].copy(), jobs[:sk].copy(),
               load.copy())
    out.hist_key, out.hist_cnt = histogram(k)
    out.qcap = (qcap_num, qcap_den)
    out.variant = variant if isinstance(variant, str) else {v: s for s, v in VARIANT.items()}[variant]
    return out


# -- f2: replanning under drift ----------------------------------------------
DIFF_FIELDS = ("keys_a", "keys_b", "keys_common", "pairs_a", "pairs_b", "pairs_common",
               "adm_k_changed", "adm_set_changed", "hist_keys", "hist_kb_changed")


def plan_kb(plan: Plan, lam: int) -> int:
    """k_b of a key with lambda requests under the plan's q_cap (Eq. 1); 1 for single-copy plans."""
    if plan.variant == "NOREPL":
        return 1
    return kb(lam, plan.qcap[0], plan.qcap[1], plan.R)


def plan_diff(a: Plan, b: Plan) -> dict:
    """Difference of two consecutive plans (supplement "Replanning Under Drift",
    replan table).  The assignment set of a plan is its set of (key, destination)
    pairs.  Count churn is over every key of either histogram, with k_b from Eq. 1
    of each plan's own rate (a key absent from a histogram has lambda = 0, k_b = 1);
    the adm_* counts compare admitted keys only (k = 0, empty set when not
    admitted).  Returns integer counts; ``churn`` turns them into the two ratios."""
    ta, tb = a.table(), b.table()
    pa = {(key, d) for key, ms in ta.items() for d in ms}
    pb = {(key, d) for key, ms in tb.items() for d in ms}
    adm = set(ta) | set(tb)
    ha = dict(zip(a.hist_key.tolist(), a.hist_cnt.tolist()))
    hb = dict(zip(b.hist_key.tolist(), b.hist_cnt.tolist()))
    hk = set(ha) | set(hb)
    return dict(
        keys_a=len(ta), keys_b=len(tb), keys_common=len(set(ta) & set(tb)),
        pairs_a=len(pa), pairs_b=len(pb), pairs_common=len(pa & pb),
        adm_k_changed=sum(1 for key in adm if len(ta.get(key, [])) != len(tb.get(key, []))),
        adm_set_changed=sum(1 for key in adm if set(ta.get(key, [])) != set(tb.get(key, []))),
        hist_keys=len(hk),
        hist_kb_changed=sum(1 for key in hk if plan_kb(a, ha.get(key, 0)) != plan_kb(b, hb.get(key, 0))))


def churn(diff: dict):
    """(cache churn, count churn) as exact fractions: cache churn = 1 - Jaccard of the two
    assignment sets; count churn = share of the keys of either histogram whose k_b changed."""
    from fractions import Fraction
    union_pairs = diff["pairs_a"] + diff["pairs_b"] - diff["pairs_common"]
    cache = 1 - Fraction(diff["pairs_common"], union_pairs) if union_pairs else Fraction(0)
    count = Fraction(diff["hist_kb_changed"], diff["hist_keys"]) if diff["hist_keys"] else Fraction(0)
    return cache, count


# -- a7 ----------------------------------------------------------------------
class Ring:
    """Consistent-hashing ring of the bounded-load policy: R destinations x V points."""

    def __init__(self, R: int, V: int, seed: int):
        self.R, self.V, self.seed = R, V, seed & ((1 << 64) - 1)
        self._h = lib().orc_ring_create(R, V, self.seed)
        if not self._h:
            raise ValueError("orc_ring_create: invalid arguments")

    def __del__(self):
        if getattr(self, "_h", None):
            lib().orc_ring_free(self._h)
            self._h = None

    def export(self):
        """(point uint64 [R*V] ascending, owner uint16 [R*V])."""
        M = self.R * self.V
        pt = np.zeros(M, np.uint64)
        ow = np.zeros(M, np.uint16)
        lib().orc_ring_export(self._h, _p(pt, C.c_uint64), _p(ow, C.c_uint16))
        return pt, ow


def route(plans: Sequence[Optional[Plan]], policies: Sequence, seeds: Sequence[int], R: int,
          keys, g0: int, B: int, load: Optional[np.ndarray] = None,
          rings: Optional[Sequence[Optional[Ring]]] = None):
    """Returns (dest uint16 [n_rep, n], load uint64 [n_rep, R])."""
    n_rep = len(policies)
    k = _c(keys, np.uint64)
    n = k.shape[0]
    pol = _c([POLICY[p] if isinstance(p, str) else p for p in policies], np.uint32)
    sd = _c(seeds, np.uint64)
    ld = np.zeros((n_rep, R), np.uint64) if load is None else _c(load, np.uint64).copy()
    dest = np.zeros((n_rep, max(n, 1)), np.uint16)
    structs = [pl._struct() if pl is not None else None for pl in plans]
    ptrs = (C.c_void_p * n_rep)(*[C.cast(C.pointer(s), C.c_void_p) if s is not None else None
                                  for s in structs])
    rg = rings if rings is not None else [None] * n_rep
    rptrs = (C.c_void_p * n_rep)(*[r._h if r is not None else None for r in rg])
    kk = k if n else np.zeros(1, np.uint64)
    rc = lib().orc_route(ptrs, rptrs, _p(pol, C.c_uint32), _p(sd, C.c_uint64), n_rep, R,
                         _p(kk, C.c_uint64), n, g0, B, _p(ld, C.c_uint64),
                         _p(dest, C.c_uint16))
    if rc != 0:
        raise ValueError(f"orc_route: status {rc}")
    return np.ascontiguousarray(dest[:, :n]), ld


# -- a8, a9 --------------------------------------------------------------------
TOKEN_LRU_MAX_ENTRIES = 1024


class Replay:
    """Whole-prefix LRU per (replica, capacity, destination); state persists across calls.
    With ``tokens`` the capacities count prefix tokens (byte-aware variant) instead of prefixes."""

    def __init__(self, n_rep: int, R: int, caps: Sequence[int], tokens: bool = False):
        self.n_rep, self.R, self.caps, self.tokens = n_rep, R, list(caps), tokens
        cp = _c(caps, np.uint32)
        make = lib().orc_replay_create_tokens if tokens else lib().orc_replay_create
        self._h = make(n_rep, R, _p(cp, C.c_uint32), len(caps))
        if not self._h:
            raise ValueError("orc_replay_create: invalid arguments")
        self.ctr = np.zeros((n_rep, len(caps), R, 5), np.uint64)

    def __del__(self):
        if getattr(self, "_h", None):
            lib().orc_replay_free(self._h)
            self._h = None

    def step(self, keys, plen, slen, dest):
        k = _c(keys, np.uint64)
        n = k.shape[0]
        if n == 0:
            return self.ctr
        p = _c(plen, np.uint32)
        s = _c(slen, np.uint32)
        d = _c(dest, np.uint16).reshape(self.n_rep, n)
        rc = lib().orc_shadow_replay(self._h, _p(k, C.c_uint64), _p(p, C.c_uint32),
                                     _p(s, C.c_uint32), _p(d, C.c_uint16), n,
                                     _p(self.ctr, C.c_uint64))
        if rc != 0:
            raise ValueError(f"orc_shadow_replay: status {rc}")
        return self.ctr

    def state(self, rep: int, cap_idx: int, r: int) -> np.ndarray:
        out = np.zeros(TOKEN_LRU_MAX_ENTRIES if self.tokens else self.caps[cap_idx], np.uint64)
        f = lib().orc_replay_state(self._h, rep, cap_idx, r, _p(out, C.c_uint64))
        return out[:f].copy()
