"""GPU parity: every CUDA kernel against the CPU oracle, element by element.

All quantities are integers, so the bar is bit-exact equality.  Inputs are
seeded synthetic traces (tracegen) or seeded random arrays; nothing the oracle
sees comes from the CUDA path.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytestmark = [pytest.mark.gpu, pytest.mark.skip(reason="needs a CUDA GPU")]
else:
    pytestmark = pytest.mark.gpu

import oracle as O
import oracle.pipeline as OP
import tracegen as tg

DEV = torch.device("cuda", 0)


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_19677_gb300 as P
    return P


@pytest.fixture(scope="module")
def ctx(P):
    c = P.Context(0)
    yield c
    c.close()


def d_u64(a):
    return torch.from_numpy(np.ascontiguousarray(a, np.uint64).view(np.int64)).to(DEV)


def d_u32(a):
    return torch.from_numpy(np.ascontiguousarray(a, np.uint32).view(np.int32)).to(DEV)


def d_u16(a):
    return torch.from_numpy(np.ascontiguousarray(a, np.uint16).view(np.int16)).to(DEV)


def h_u64(t):
    return t.cpu().numpy().view(np.uint64)


def h_u16(t):
    return t.cpu().numpy().view(np.uint16)


# ------------------------------------------------------------------ a1 hash ---
@pytest.mark.parametrize("align", [1, 2, 4])
def test_hash_trace(P, ctx, align):
    cfg = tg.CONFIGS["70b"].scaled(3000, 1)
    tr = tg.Trace(cfg)
    iv = tr.interval(0)
    tok, off = tg.arena_host(tr, iv, align)
    ref = O.hash_prefixes(tok, off, iv.plen, salt=12345)
    got = P.hash_prefixes(ctx, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), salt=12345)
    ctx.sync()
    assert (h_u64(got) == ref).all()


def test_hash_edge_lengths_and_offsets(P, ctx):
    rng = np.random.default_rng(5)
    lens = [0, 1, 2, 3, 4, 5, 7, 8, 9, 63, 64, 65, 127, 128, 129, 255, 256, 257, 511, 512, 513, 1023,
            1024, 1025, 4095, 4096, 4097, 16383, 16384, 32768]
    tok = rng.integers(-2**31, 2**31, size=200_000, dtype=np.int64).astype(np.int32)
    offs, plens = [], []
    for o0 in range(8):               # every alignment of the span start
        for L in lens:
            o = int(rng.integers(0, tok.size - L - 8)) // 8 * 8 + o0
            offs.append(o)
            plens.append(L)
    offs = np.array(offs, np.uint64)
    plens = np.array(plens, np.uint32)
    ref = O.hash_prefixes(tok, offs, plens, salt=(1 << 64) - 3)
    got = P.hash_prefixes(ctx, torch.from_numpy(tok).to(DEV), d_u64(offs), d_u32(plens), salt=(1 << 64) - 3)
    ctx.sync()
    assert (h_u64(got) == ref).all()


def test_hash_empty(P, ctx):
    t = torch.zeros(4, dtype=torch.int32, device=DEV)
    out = P.hash_prefixes(ctx, t, torch.zeros(0, dtype=torch.int64, device=DEV),
                          torch.zeros(0, dtype=torch.int32, device=DEV))
    ctx.sync()
    assert out.numel() == 0


# ------------------------------------------------------------------ a2..a6 ---
def _rates_keys(rng, nkeys, total, skew=1.2):
    w = rng.pareto(skew, size=nkeys) + 1e-3
    c = np.maximum(1, np.round(w / w.sum() * total)).astype(np.int64)
    ks = rng.integers(0, 2**64, size=nkeys, dtype=np.uint64)
    keys = np.repeat(ks, c)
    rng.shuffle(keys)
    return keys


def _cmp_plan(got, ref):
    assert got["U"] == ref.U
    assert got["n_adm"] == ref.n_adm and got["sum_k"] == ref.sum_k and got["cold"] == ref.cold
    assert (got["adm_key"] == ref.adm_key).all()
    assert (got["adm_cnt"] == ref.adm_cnt).all()
    assert (got["adm_k"] == ref.adm_k).all()
    assert (got["koff"] == ref.koff).all()
    assert (got["members"] == ref.members).all()
    assert (got["jobs"] == ref.jobs).all()
    assert (got["load"] == ref.load).all()


@pytest.mark.parametrize("seed", range(8))
def test_plan_parity(P, ctx, seed):
    rng = np.random.default_rng(200 + seed)
    R = int(rng.choice([1, 2, 3, 7, 30, 64, 100, 1024]))
    W = int(rng.integers(1, 20))
    nkeys = int(rng.integers(1, 5000))
    keys = _rates_keys(rng, nkeys, int(rng.integers(nkeys, 60000)))
    n = keys.size
    num, den = (5 * n, 4 * R) if seed % 2 == 0 else (n, 9 * R)
    variants = ("LPT", "RANDOM", "NOREPL", "SLOTCAP")
    plans = [P.Plan(ctx) for _ in variants]
    params = [P.plan_params(R, W, num, den, v, seed=seed, epoch=3) for v in variants]
    P.build_plans(ctx, d_u64(keys), params, plans)
    uk, uc = O.histogram(keys)
    for pl, v in zip(plans, variants):
        got = pl.export()
        assert (got["ukey"] == uk).all() and (got["ucnt"] == uc).all()
        _cmp_plan(got, O.build_plan(keys, R, W, num, den, variant=v, seed=seed, epoch=3))


def _keys_with_counts(rng, counts):
    ks = np.unique(rng.integers(0, 2**64 - 1, size=len(counts) + 64, dtype=np.uint64))[:len(counts)]
    rng.shuffle(ks)
    keys = np.repeat(ks, np.asarray(counts, np.int64))
    rng.shuffle(keys)
    return keys


@pytest.mark.parametrize("case", ["ties_at_threshold", "U_eq_C", "U_eq_C_minus_1", "U_eq_C_plus_1",
                                  "wide_counts", "single_key", "all_equal"])
def test_plan_admission_candidates(P, ctx, case):
    # the planner sorts only keys whose count reaches the C-th largest (C = R*W);
    # these traces put that threshold on its edge cases
    rng = np.random.default_rng(len(case))
    R, W = 8, 5                      # C = 40
    if case == "ties_at_threshold":  # 30 distinct counts above, 500 keys tied at the 40th count
        counts = list(range(100, 130)) + [7] * 500 + [3] * 200
    elif case == "U_eq_C":
        counts = list(rng.integers(1, 50, size=40))
    elif case == "U_eq_C_minus_1":
        counts = list(rng.integers(1, 50, size=39))
    elif case == "U_eq_C_plus_1":
        counts = list(rng.integers(1, 50, size=41))
    elif case == "wide_counts":      # counts over 17 bits: both select levels matter
        counts = list(rng.integers(1, 120000, size=60)) + list(rng.integers(1, 40, size=3000))
    elif case == "single_key":
        R, W = 1, 1
        counts = [12345]
    else:                            # every key ties
        counts = [5] * 2000
    keys = _keys_with_counts(rng, counts)
    n = keys.size
    params = [P.plan_params(R, W, 5 * n, 4 * R, v, seed=2, epoch=4) for v in ("LPT", "RANDOM", "NOREPL")]
    plans = [P.Plan(ctx) for _ in params]
    P.build_plans(ctx, d_u64(keys), params, plans)
    uk, uc = O.histogram(keys)
    for pl, v in zip(plans, ("LPT", "RANDOM", "NOREPL")):
        got = pl.export()
        assert (got["ukey"] == uk).all() and (got["ucnt"] == uc).all()
        _cmp_plan(got, O.build_plan(keys, R, W, 5 * n, 4 * R, variant=v, seed=2, epoch=4))


@pytest.mark.parametrize("R,nkeys,total", [(30, 150000, 400000), (1024, 300000, 1200000)])
def test_plan_parity_large_histogram(P, ctx, R, nkeys, total):
    # histograms far above the one-CTA sort size (device-wide radix passes)
    rng = np.random.default_rng(nkeys)
    keys = _rates_keys(rng, nkeys, total, skew=0.9)
    n = keys.size
    params = [P.plan_params(R, 64, 5 * n, 4 * R, v, seed=3, epoch=1) for v in ("LPT", "RANDOM", "NOREPL")]
    plans = [P.Plan(ctx) for _ in params]
    P.build_plans(ctx, d_u64(keys), params, plans)
    uk, uc = O.histogram(keys)
    for pl, v in zip(plans, ("LPT", "RANDOM", "NOREPL")):
        got = pl.export()
        assert (got["ukey"] == uk).all() and (got["ucnt"] == uc).all()
        _cmp_plan(got, O.build_plan(keys, R, 64, 5 * n, 4 * R, variant=v, seed=3, epoch=1))


@pytest.mark.parametrize("R,spread", [(33, 0), (64, 50), (257, 3), (1024, 0), (1024, 400)])
def test_plan_equal_rate_runs(P, ctx, R, spread):
    # long runs of keys with the same count and k = 1 (placed a run at a time on
    # the device), hot replicated keys before them, short runs, runs with
    # counts above 1024, and uneven starting loads
    rng = np.random.default_rng(R + spread)
    counts = [3000] * 2 + [1500] * 3 + [1100] * 40 + [37] * 70 + [5] * 300 + [2] * 900 + [1] * 5000
    counts += list(rng.integers(1, 60, size=200))
    ks = np.unique(rng.integers(0, 2**64 - 1, size=len(counts) + 64, dtype=np.uint64))[:len(counts)]
    rng.shuffle(ks)
    keys = np.repeat(ks, counts)
    rng.shuffle(keys)
    init = None
    if spread:
        init = rng.integers(0, spread + 1, size=R).astype(np.uint64)
    W = 2 + 6500 // R
    params = [P.plan_params(R, W, 2000, 1, v, init_load=None if init is None else d_u64(init))
              for v in ("LPT", "NOREPL")]
    plans = [P.Plan(ctx) for _ in params]
    P.build_plans(ctx, d_u64(keys), params, plans)
    for pl, v in zip(plans, ("LPT", "NOREPL")):
        _cmp_plan(pl.export(), O.build_plan(keys, R, W, 2000, 1, variant=v, init_load=init))


def test_plan_hand_example_and_init_load(P, ctx):
    keys = np.array([1] * 21 + [2] * 6 + [3] * 3 + [4], np.uint64)
    pl = P.build_plan(ctx, d_u64(keys), P.plan_params(3, 1, 155, 12))
    _cmp_plan(pl.export(), O.build_plan(keys, 3, 1, 155, 12))
    init = np.array([9, 0, 4], np.uint64)
    pl2 = P.build_plan(ctx, d_u64(keys), P.plan_params(3, 2, 1000, 1, init_load=d_u64(init)))
    _cmp_plan(pl2.export(), O.build_plan(keys, 3, 2, 1000, 1, init_load=init))


@pytest.mark.parametrize("extra", [[2**64 - 1], [0], [2**64 - 1, 0, 2**64 - 1, 2**64 - 2]])
def test_plan_extreme_keys(P, ctx, extra):
    # the all-ones key doubles as the device table's empty marker and is counted apart
    rng = np.random.default_rng(len(extra))
    keys = np.concatenate([_rates_keys(rng, 500, 5000), np.array(extra * 7, np.uint64)])
    rng.shuffle(keys)
    R, W = 8, 4
    pl = P.build_plan(ctx, d_u64(keys), P.plan_params(R, W, keys.size, 3 * R))
    got = pl.export()
    uk, uc = O.histogram(keys)
    assert (got["ukey"] == uk).all() and (got["ucnt"] == uc).all()
    _cmp_plan(got, O.build_plan(keys, R, W, keys.size, 3 * R))


def test_plan_empty_and_single(P, ctx):
    pl = P.build_plan(ctx, torch.zeros(0, dtype=torch.int64, device=DEV), P.plan_params(4, 2, 1, 1))
    got = pl.export()
    assert got["U"] == 0 and got["n_adm"] == 0 and (got["load"] == 0).all()
    keys = np.array([7, 7, 7], np.uint64)
    pl = P.build_plan(ctx, d_u64(keys), P.plan_params(5, 1, 1, 1))   # q_cap = 1: k = min(R, 3)
    _cmp_plan(pl.export(), O.build_plan(keys, 5, 1, 1, 1))


def test_plan_bad_params(P, ctx):
    keys = d_u64(np.array([1, 2], np.uint64))
    with pytest.raises(P.CacheRouteError):
        P.build_plan(ctx, keys, P.plan_params(0, 1, 1, 1))
    with pytest.raises(P.CacheRouteError):
        P.build_plan(ctx, keys, P.plan_params(4, 1, 1, 0))
    with pytest.raises(P.CacheRouteError):
        P.build_plan(ctx, keys, P.plan_params(P.MAX_R + 1, 1, 1, 1))


# ------------------------------------------------------------------ a7 route ---
@pytest.mark.parametrize("R,B", [(1, 1), (3, 1), (7, 33), (30, 1024), (64, 5000), (1024, 256), (30, 20000),
                                 (5, 16384), (9, 16385), (1024, 1), (64, 2), (30, 3), (7, 31), (1024, 32),
                                 (257, 5), (8192, 1), (8192, 7), (8192, 64)])
def test_route_parity(P, ctx, R, B):
    # batches of <= 32 requests take the one-warp-per-replica kernel, longer ones the CTA kernel
    rng = np.random.default_rng(R * 7 + B)
    keys = _rates_keys(rng, 3000, 40000)
    n = keys.size
    pols = ["CR", "CR_NOLPT", "CR_NOREPL", "P2C", "RR", "HASH", "CR", "P2C", "CHWBL", "CHWBL"]
    seeds = [0, 1, 0, 2, 3, 4, 9, 2**63 + 5, 11, 2**64 - 1]
    ring_args = {8: (64, 5), 9: (1, 2**63 + 1)}  # replica -> (vnodes, ring seed)
    orings = [O.Ring(R, *ring_args[i]) if i in ring_args else None for i in range(len(pols))]
    drings = [P.Ring(ctx, R, *ring_args[i]) if i in ring_args else None for i in range(len(pols))]
    num, den = n, 6 * R            # tight: replicated keys
    W = 4
    oplans = {v: O.build_plan(keys, R, W, num, den, variant=v, seed=s, epoch=1)
              for v, s in (("LPT", 0), ("RANDOM", 1), ("NOREPL", 0))}
    dplans = {}
    for v, s in (("LPT", 0), ("RANDOM", 1), ("NOREPL", 0)):
        dplans[v] = P.build_plan(ctx, d_u64(keys), P.plan_params(R, W, num, den, v, seed=s, epoch=1))
    vmap = {"CR": "LPT", "CR_NOLPT": "RANDOM", "CR_NOREPL": "NOREPL"}
    init = rng.integers(0, 50, size=(len(pols), R)).astype(np.uint64)
    ref_dest, ref_load = O.route([oplans.get(vmap.get(p)) for p in pols], pols, seeds, R, keys, 777, B,
                                 load=init, rings=orings)
    load = d_u64(init.reshape(-1)).view(len(pols), R).contiguous()
    dest = P.route_batch(ctx, [dplans.get(vmap.get(p)) for p in pols], pols, seeds, R, d_u64(keys), 777, B, load,
                         rings=drings)
    ctx.sync()
    for i, p in enumerate(pols):
        assert (h_u16(dest[i]) == ref_dest[i]).all(), (i, p)
    assert (h_u64(load) == ref_load).all()


@pytest.mark.parametrize("R", [1, 30, 1024, 8191])
@pytest.mark.parametrize("g0,seed", [(0, 2**64 - 1000), (2**40 + 3, 2**64 - 2**40 - 2500), (2**33, 7), (0, 0)])
def test_route_rr_hash_index_edges(P, ctx, R, g0, seed):
    # round robin is (g0 + i + seed) mod 2^64 mod R: the sum wraps inside the call for the
    # first two seeds, and request indices start above 2^32 for the second and third
    rng = np.random.default_rng(R)
    keys = rng.integers(0, 2**63, 5000, dtype=np.int64).astype(np.uint64)
    pols, seeds = ["RR", "HASH", "P2C"], [seed, seed ^ 5, seed]
    ref_dest, ref_load = O.route([None] * 3, pols, seeds, R, keys, g0, 1024)
    load = torch.zeros((3, R), dtype=torch.int64, device=DEV)
    dest = P.route_batch(ctx, [None] * 3, pols, seeds, R, d_u64(keys), g0, 1024, load)
    ctx.sync()
    for i, p in enumerate(pols):
        assert (h_u16(dest[i]) == ref_dest[i]).all(), p
    assert (h_u64(load) == ref_load).all()


@pytest.mark.parametrize("R,V,seed", [(1, 1, 0), (3, 1, 0), (7, 5, 123), (1024, 64, 9), (8192, 16, 2**64 - 1),
                                      (5, 1024, 77)])
def test_ring_parity(P, ctx, R, V, seed):
    pt, ow = P.Ring(ctx, R, V, seed).export()
    opt, oow = O.Ring(R, V, seed).export()
    assert (pt == opt).all() and (ow == oow).all()


def _inv_mix(z):
    m64 = (1 << 64) - 1

    def unxs(y, s):
        x = y
        for _ in range(64 // s + 1):
            x = y ^ (x >> s)
        return x & m64
    z = unxs(z, 31)
    z = (z * pow(0x94D049BB133111EB, -1, 1 << 64)) & m64
    z = unxs(z, 27)
    z = (z * pow(0xBF58476D1CE4E5B9, -1, 1 << 64)) & m64
    return unxs(z, 30)


@pytest.mark.parametrize("R,V,B", [(2, 1, 1), (13, 3, 1), (13, 3, 4), (600, 8, 1), (600, 8, 1000)])
def test_route_chwbl_ring_edges(P, ctx, R, V, B):
    # keys exactly on ring points, one past a point, past the last point (wrap), on a
    # half-saturated fleet, so walks run past destinations at their bound
    rng = np.random.default_rng(R + B)
    rs, ks = 2**62 + R, 12345
    opt, _ = O.Ring(R, V, rs).export()
    edge = []
    for p in [int(x) for x in opt[:4]] + [int(x) for x in opt[-4:]]:
        edge += [_inv_mix(p) ^ ks, _inv_mix((p + 1) % 2**64) ^ ks]
    edge += [_inv_mix(2**64 - 1) ^ ks, _inv_mix(0) ^ ks]
    hot = rng.integers(0, 2**63, 8, dtype=np.int64).astype(np.uint64)
    keys = np.concatenate([np.array(edge, np.uint64), hot[rng.integers(0, 8, 5000)],
                           rng.integers(0, 2**63, 3000, dtype=np.int64).astype(np.uint64)])
    rng.shuffle(keys)
    init = np.zeros((1, R), np.uint64)
    init[0, : R // 2] = rng.integers(0, 30, R // 2).astype(np.uint64) + np.uint64(keys.size // R)
    ref_dest, ref_load = O.route([None], ["CHWBL"], [ks], R, keys, 5, B, load=init, rings=[O.Ring(R, V, rs)])
    load = d_u64(init.reshape(-1)).view(1, R).contiguous()
    dest = P.route_batch(ctx, [None], ["CHWBL"], [ks], R, d_u64(keys), 5, B, load, rings=[P.Ring(ctx, R, V, rs)])
    ctx.sync()
    assert (h_u16(dest) == ref_dest).all()
    assert (h_u64(load) == ref_load).all()


@pytest.mark.parametrize("B", [1, 2, 3, 16, 32])
def test_route_small_batches_one_hot_key(P, ctx, B):
    # every request carries the same replicated key: every lane of a warp step competes
    # for the same members, the slowest case of the fixed-point resolution
    R, W = 64, 2
    keys = np.concatenate([np.full(20000, 0xDEADBEEF, np.uint64), np.arange(1, 2001, dtype=np.uint64)])
    num, den = 1, 1  # q_cap = 1: k_b = min(R, lambda) -> all R destinations
    opl = O.build_plan(keys, R, W, num, den)
    dpl = P.build_plan(ctx, d_u64(keys), P.plan_params(R, W, num, den))
    pols, seeds = ["CR", "P2C", "CHWBL"], [0, 1, 2]
    ref_dest, ref_load = O.route([opl, None, None], pols, seeds, R, keys, 0, B,
                                 rings=[None, None, O.Ring(R, 4, 3)])
    load = torch.zeros((3, R), dtype=torch.int64, device=DEV)
    dest = P.route_batch(ctx, [dpl, None, None], pols, seeds, R, d_u64(keys), 0, B, load,
                         rings=[None, None, P.Ring(ctx, R, 4, 3)])
    ctx.sync()
    assert (h_u16(dest) == ref_dest).all()
    assert (h_u64(load) == ref_load).all()


@pytest.mark.parametrize("case", ["few", "many", "pool", "wide"])
@pytest.mark.parametrize("B", [100, 1024])
def test_route_replicated_keys_per_batch(P, ctx, case, B):
    # keys with k_b > 1 decided once per batch from a shared-memory cache of their member
    # lists: a few such keys; more keys than the cache holds (300); member lists larger than
    # its pool (two keys on every one of 4096 destinations); and R = 8192, where the cache
    # does not fit beside the loads.  q_cap = 1, so a key seen c times gets k_b = min(c, R).
    rng = np.random.default_rng(B + len(case))
    R, W = {"few": (64, 64), "many": (64, 64), "pool": (4096, 2), "wide": (8192, 1)}[case]
    counts = {"few": [2, 3, 5, 8, 13, 21, 34, 55, 64, 64], "many": [2] * 300 + [3] * 20,
              "pool": [4096, 4096], "wide": [7, 300, 2]}[case]
    ks = rng.integers(1, 2**63, len(counts) + 30000, dtype=np.int64).astype(np.uint64)
    keys = np.concatenate([np.repeat(ks[: len(counts)], counts), ks[len(counts):]])
    rng.shuffle(keys)
    pols, seeds = ["CR", "CR_NOLPT", "CR_NOREPL", "P2C", "CR"], [0, 1, 0, 2, 3]
    vmap = {"CR": ("LPT", 0), "CR_NOLPT": ("RANDOM", 1), "CR_NOREPL": ("NOREPL", 0)}
    opl = {p: O.build_plan(keys, R, W, 1, 1, variant=v, seed=s, epoch=0) for p, (v, s) in vmap.items()}
    dpl = {p: P.build_plan(ctx, d_u64(keys), P.plan_params(R, W, 1, 1, v, seed=s, epoch=0))
           for p, (v, s) in vmap.items()}
    assert (np.asarray(opl["CR"].adm_k) > 1).sum() >= min(len(counts), 2)
    init = rng.integers(0, 9, size=(len(pols), R)).astype(np.uint64)
    ref_dest, ref_load = O.route([opl.get(p) for p in pols], pols, seeds, R, keys, 11, B, load=init)
    load = d_u64(init.reshape(-1)).view(len(pols), R).contiguous()
    dest = P.route_batch(ctx, [dpl.get(p) for p in pols], pols, seeds, R, d_u64(keys), 11, B, load)
    ctx.sync()
    for i, p in enumerate(pols):
        assert (h_u16(dest[i]) == ref_dest[i]).all(), (i, p)
    assert (h_u64(load) == ref_load).all()


def test_route_rejects_bad_args(P, ctx):
    keys = d_u64(np.array([1, 2, 3], np.uint64))
    load = torch.zeros((1, 4), dtype=torch.int64, device=DEV)
    with pytest.raises(P.CacheRouteError):
        P.route_batch(ctx, [None], ["CR"], [0], 4, keys, 0, 16, load)       # plan missing
    with pytest.raises(P.CacheRouteError):
        P.route_batch(ctx, [None], ["P2C"], [0], 4, keys, 0, 0, load)       # B = 0
    with pytest.raises(P.CacheRouteError):
        P.route_batch(ctx, [None], ["P2C"], [0], 0, keys, 0, 4, load)       # R = 0
    with pytest.raises(P.CacheRouteError):
        P.route_batch(ctx, [None], ["CHWBL"], [0], 4, keys, 0, 1, load)     # ring missing
    with pytest.raises(P.CacheRouteError):
        P.route_batch(ctx, [None], ["CHWBL"], [0], 4, keys, 0, 1, load, rings=[P.Ring(ctx, 5, 2, 0)])  # R differs
    with pytest.raises(P.CacheRouteError):
        P.Ring(ctx, 4, 0, 0)                                                # no points
    with pytest.raises(P.CacheRouteError):
        P.Ring(ctx, 4, P.MAX_VNODES + 1, 0)


# ------------------------------------------------------------------ a8, a9 ---
@pytest.mark.parametrize("caps", [[1], [2, 16], [12], [32], [33], [64, 256, 1024], [5, 33, 100], [1024],
                                  [1, 40, 64], [2, 2, 50], [256, 64], [1, 2, 3, 4, 5, 6, 7, 40]])
def test_replay_parity(P, ctx, caps):
    rng = np.random.default_rng(sum(caps))
    n_rep, R = 3, 5
    n = 20000
    keys = _rates_keys(rng, int(rng.integers(20, 3000)), n)[:n]
    n = keys.size
    plen = rng.integers(16, 5000, size=n).astype(np.uint32)
    slen = np.full(n, 64, np.uint32)
    dest = tg.random_dest(n_rep, n, R, 3)
    orp = O.Replay(n_rep, R, caps)
    rp = P.Replay(ctx, n_rep, R, caps)
    ctr = torch.zeros((n_rep, len(caps), R, 5), dtype=torch.int64, device=DEV)
    dk, dp, ds, dd = d_u64(keys), d_u32(plen), d_u32(slen), d_u16(dest)
    # two calls: state persists across them
    cut = n // 3
    for a, b in ((0, cut), (cut, n)):
        orp.step(keys[a:b], plen[a:b], slen[a:b], dest[:, a:b])
        P.shadow_replay(ctx, rp, dk[a:b].contiguous(), dp[a:b].contiguous(), ds[a:b].contiguous(),
                        dd[:, a:b].contiguous(), ctr)
        ctx.sync()
        assert (h_u64(ctr) == orp.ctr).all()
    cmax = max(caps)
    for rep in range(n_rep):
        for r in range(R):
            st = rp.state(rep, r)
            ci = caps.index(cmax)
            assert (st == orp.state(rep, ci, r)).all()
            for c_i, c in enumerate(caps):
                assert (st[:c] == orp.state(rep, c_i, r)).all()


@pytest.mark.parametrize("nkeys", [1500, 6000])
def test_replay_parity_long_streams(P, ctx, nkeys):
    # streams far longer than any chunk the replay splits work into (> 16,384 requests per
    # stream per call), at the Large configuration's capacities: the state each chunk starts
    # from must be rebuilt exactly, in both calls (the second starts from persisted state)
    rng = np.random.default_rng(nkeys)
    caps = [64, 256, 1024]
    n_rep, R = 2, 2
    keys = _rates_keys(rng, nkeys, 130000, skew=0.9)
    n = keys.size
    plen = rng.integers(16, 5000, size=n).astype(np.uint32)
    slen = np.full(n, 64, np.uint32)
    dest = tg.random_dest(n_rep, n, R, 11)
    orp = O.Replay(n_rep, R, caps)
    rp = P.Replay(ctx, n_rep, R, caps)
    ctr = torch.zeros((n_rep, len(caps), R, 5), dtype=torch.int64, device=DEV)
    dk, dp, ds, dd = d_u64(keys), d_u32(plen), d_u32(slen), d_u16(dest)
    cut = n // 3
    for a, b in ((0, cut), (cut, n)):
        per_stream = np.bincount(dest[0, a:b], minlength=R)
        assert per_stream.min() > 16384
        orp.step(keys[a:b], plen[a:b], slen[a:b], dest[:, a:b])
        P.shadow_replay(ctx, rp, dk[a:b].contiguous(), dp[a:b].contiguous(), ds[a:b].contiguous(),
                        dd[:, a:b].contiguous(), ctr)
        ctx.sync()
        got = h_u64(ctr)
        assert (got == orp.ctr).all()
        assert 0 < got[:, 0, :, 1].sum() < got[:, 2, :, 1].sum() < got[:, 2, :, 0].sum()  # hits differ by cap
    for rep in range(n_rep):
        for r in range(R):
            st = rp.state(rep, r)
            for c_i, c in enumerate(caps):
                assert (st[:c] == orp.state(rep, c_i, r)).all()


def test_replay_reset_and_bad_dest(P, ctx):
    rp = P.Replay(ctx, 1, 4, [8])
    keys = d_u64(np.arange(10, dtype=np.uint64))
    plen = d_u32(np.full(10, 5, np.uint32))
    dest = d_u16(np.array([[0, 1, 2, 3, 0, 1, 2, 3, 0, 9]], np.uint16))   # 9 >= R
    ctr = torch.zeros((1, 1, 4, 5), dtype=torch.int64, device=DEV)
    P.shadow_replay(ctx, rp, keys, plen, plen, dest, ctr)
    with pytest.raises(P.CacheRouteError):
        ctx.sync()
    assert int(ctr[..., 0].sum()) == 9
    rp.reset()
    ctx.sync()
    assert rp.state(0, 0).size == 0


# ------------------------------------------------------------------ pipeline ---
@pytest.mark.parametrize("overlap", [False, True])
@pytest.mark.parametrize("name,n,nint", [("tiny", 20000, 1), ("70b", 30000, 3), ("8b", 6000, 4),
                                          ("burst", 30000, 2), ("70b-gamma", 30000, 3)])
def test_pipeline_parity(P, ctx, name, n, nint, overlap):
    from paper_2608_19677_gb300.pipeline import Pipeline
    cfg = tg.CONFIGS[name]
    if name != "tiny":
        cfg = cfg.scaled(n, nint)
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=1024, keep=True)
    pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=1024, overlap=overlap)
    for rep in range(2):          # twice: reset() must restore the initial state
        pipe.reset()
        for t in range(cfg.n_intervals):
            iv = tr.interval(t)
            tok, off = tg.arena_host(tr, iv, 4)
            keys = pipe.interval(t, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), d_u32(iv.slen),
                                 iv.g0, plan_next=t + 1 < cfg.n_intervals)
            assert (h_u64(keys) == ref["keys"][t]).all()
            pipe.wait_last()
            assert (h_u16(pipe.last_dest) == ref["dest"][t]).all()
            # the plans the interval was routed with equal the oracle's
            for (v, s), pl in zip(pipe.plan_keys, pipe.last_plans):
                opl = ref["plans"][t][(v, s)]
                got = pl.export()
                assert got["n_adm"] == opl.n_adm and (got["members"] == opl.members).all()
        pipe.sync()
        assert (h_u64(pipe.ctr) == ref["ctr"]).all()


@pytest.mark.parametrize("name,n,nint,depth,ps,rs,grp", [("70b", 40000, 6, 3, 2, 2, 1), ("8b", 8000, 9, 4, 3, 2, 1),
                                                          ("burst", 40000, 4, 2, 1, 3, 1),
                                                          ("large", 200000, 3, 8, 4, 4, 1),
                                                          ("tiny", 20000, 1, 8, 4, 4, 1),
                                                          ("70b", 40000, 7, 4, 2, 3, 3), ("8b", 8000, 9, 6, 2, 2, 4),
                                                          ("large", 200000, 3, 8, 4, 4, 2)])
def test_trace_pipeline_parity(P, ctx, name, n, nint, depth, ps, rs, grp):
    # several intervals in flight (plans and routes on several streams, the replay in order):
    # every interval's plans and destinations, and the counters, equal the oracle's
    from paper_2608_19677_gb300.pipeline import TracePipeline
    cfg = tg.CONFIGS[name]
    if name != "tiny":
        cfg = cfg.scaled(n, nint)
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=1024, keep=True)
    ivs = [tr.interval(t) for t in range(cfg.n_intervals)]
    keys = [d_u64(k) for k in ref["keys"]]
    plens = [d_u32(iv.plen) for iv in ivs]
    slens = [d_u32(iv.slen) for iv in ivs]
    pipe = TracePipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, max_n=max(iv.n for iv in ivs),
                         batch_B=1024, depth=depth, plan_streams=ps, route_streams=rs, vnodes=cfg.vnodes,
                         replay_group=grp)
    for rep in range(2):   # twice: reset() restores the initial state
        pipe.reset()
        seen = []

        def check(t, dest, plans):
            pipe.sync()
            seen.append(t)
            assert (h_u16(dest) == ref["dest"][t]).all(), f"interval {t}: destinations differ"
            for (v, s_), pl in zip(pipe.plan_keys, plans):
                opl = ref["plans"][t][(v, s_)]
                got = pl.export()
                assert got["n_adm"] == opl.n_adm and (got["members"] == opl.members).all()
        pipe.run(keys, plens, slens, [iv.g0 for iv in ivs], on_interval=check if rep == 0 else None)
        pipe.sync()
        assert (h_u64(pipe.ctr) == ref["ctr"]).all()
    pipe.close()


@pytest.mark.parametrize("name,grp", [("8b", 4), ("70b", 2)])
def test_trace_pipeline_cuda_graph(P, ctx, name, grp):
    # the whole trace (reset + every interval's plans, routes and replay, on many streams)
    # captured once as a CUDA graph: each replay gives the oracle's counters again
    from paper_2608_19677_gb300.pipeline import TracePipeline
    cfg = tg.CONFIGS[name].scaled(40000, 8)
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=1024, keep=True)
    ivs = [tr.interval(t) for t in range(cfg.n_intervals)]
    keys = [d_u64(k) for k in ref["keys"]]
    plens = [d_u32(iv.plen) for iv in ivs]
    slens = [d_u32(iv.slen) for iv in ivs]
    g0s = [iv.g0 for iv in ivs]
    stream = torch.cuda.Stream()       # a graph is captured on a stream other than the default one
    gctx = P.Context(0, stream)
    pipe = TracePipeline(gctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, max_n=max(iv.n for iv in ivs),
                         batch_B=1024, depth=4, plan_streams=3, route_streams=2, vnodes=cfg.vnodes,
                         replay_group=grp)
    pipe.reset()
    pipe.run(keys, plens, slens, g0s)   # warm-up: scratch and inputs reach their sizes
    pipe.quiesce()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        pipe.reset()
        pipe.run(keys, plens, slens, g0s)
    for _ in range(2):
        graph.replay()
        torch.cuda.synchronize()
        assert (h_u64(pipe.ctr) == ref["ctr"]).all()
    del graph
    pipe.close()
    gctx.close()


@pytest.mark.parametrize("B", [1, 7, 1024])
def test_pipeline_parity_bounded_load_and_small_batches(P, ctx, B):
    # the 70B shape with the bounded-load comparison policy added, routed in
    # batches of 1 (exact sequential), 7 and 1024 requests
    import dataclasses
    from paper_2608_19677_gb300.pipeline import Pipeline
    cfg = dataclasses.replace(tg.CONFIGS["70b"].scaled(20000, 2), policies=["CR", "P2C", "HASH", "CHWBL"],
                              seeds=[0, 3])
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=B, keep=True)
    pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=B, overlap=True,
                    vnodes=cfg.vnodes)
    for t in range(cfg.n_intervals):
        iv = tr.interval(t)
        tok, off = tg.arena_host(tr, iv, 4)
        pipe.interval(t, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), d_u32(iv.slen), iv.g0,
                      plan_next=t + 1 < cfg.n_intervals)
        pipe.wait_last()
        assert (h_u16(pipe.last_dest) == ref["dest"][t]).all()
    pipe.sync()
    assert (h_u64(pipe.ctr) == ref["ctr"]).all()


# ------------------------------------------------------------------ f2 replanning ---
def _diff_case(P, ctx, keys_a, keys_b, R, W, num_den_a, num_den_b, var_a="LPT", var_b="LPT"):
    oa = O.build_plan(keys_a, R, W, *num_den_a, variant=var_a, seed=1, epoch=0)
    ob = O.build_plan(keys_b, R, W, *num_den_b, variant=var_b, seed=2, epoch=1)
    da = P.build_plan(ctx, d_u64(keys_a), P.plan_params(R, W, *num_den_a, var_a, seed=1, epoch=0))
    db = P.build_plan(ctx, d_u64(keys_b), P.plan_params(R, W, *num_den_b, var_b, seed=2, epoch=1))
    got = P.plan_diff(ctx, da, db)
    want = O.plan_diff(oa, ob)
    assert got == want
    assert P.plan_diff(ctx, db, da) == O.plan_diff(ob, oa)
    assert P.plan_diff(ctx, da, da) == O.plan_diff(oa, oa)
    return got


@pytest.mark.parametrize("t", range(5))
def test_plan_diff_drift_transitions(P, ctx, t):
    # consecutive fresh LPT plans of the drift trace (70B shape, lognormal rate walk)
    cfg = tg.CONFIGS["drift"]
    tr = tg.Trace(cfg)
    ka = O.hash_prefixes(*tg.arena_host(tr, tr.interval(t), 4), tr.interval(t).plen)
    kb = O.hash_prefixes(*tg.arena_host(tr, tr.interval(t + 1), 4), tr.interval(t + 1).plen)
    d = _diff_case(P, ctx, ka, kb, cfg.R, cfg.W, tr.qcap(ka.size), tr.qcap(kb.size))
    cache, count = O.churn(d)
    assert 0 < cache <= 1 and 0 <= count < 1


@pytest.mark.parametrize("R,W,spread", [(1, 4, 50), (7, 3, 400), (64, 8, 3000), (1024, 16, 20000),
                                        (8192, 2, 30000)])
def test_plan_diff_shapes(P, ctx, R, W, spread):
    rng = np.random.default_rng(R)
    ka = _rates_keys(rng, spread, 60000)
    kb = np.concatenate([ka[: ka.size // 2], _rates_keys(rng, spread, 30000)])  # half the traffic changes
    n = ka.size
    _diff_case(P, ctx, ka, kb, R, W, (n, 4 * R), (n, 3 * R), "LPT", "RANDOM")  # replicated keys, k_b up to R


def test_plan_diff_empty_and_errors(P, ctx):
    keys = np.arange(1, 500, dtype=np.uint64) * np.uint64(7919)
    e = np.zeros(0, np.uint64)
    _diff_case(P, ctx, e, keys, 16, 4, (1, 1), (keys.size, 64))
    _diff_case(P, ctx, e, e, 16, 4, (1, 1), (1, 1))
    a = P.build_plan(ctx, d_u64(keys), P.plan_params(16, 4, keys.size, 64))
    b = P.build_plan(ctx, d_u64(keys), P.plan_params(17, 4, keys.size, 64))
    with pytest.raises(P.CacheRouteError):
        P.plan_diff(ctx, a, b)                                              # R differs
    with pytest.raises(P.CacheRouteError):
        P.plan_diff(ctx, a, P.Plan(ctx))                                    # not built


@pytest.mark.parametrize("fresh", [True, False])
def test_pipeline_parity_drift_fresh_and_stale(P, ctx, fresh):
    # the replanning comparison: every interval routed with a plan from its own keys
    # (fresh) or from the previous interval's (stale), replayed through persistent LRUs
    from paper_2608_19677_gb300.pipeline import Pipeline
    cfg = tg.CONFIGS["drift"].scaled(60000, 6)
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=1024, keep=True, fresh=fresh)
    pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=1024, overlap=True, fresh=fresh)
    for t in range(cfg.n_intervals):
        iv = tr.interval(t)
        tok, off = tg.arena_host(tr, iv, 4)
        pipe.interval(t, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), d_u32(iv.slen), iv.g0,
                      plan_next=t + 1 < cfg.n_intervals)
        pipe.wait_last()
        assert (h_u16(pipe.last_dest) == ref["dest"][t]).all()
        for (v, s), pl in zip(pipe.plan_keys, pipe.last_plans):
            got = pl.export()
            opl = ref["plans"][t][(v, s)]
            assert got["n_adm"] == opl.n_adm and (got["members"] == opl.members).all()
    pipe.sync()
    assert (h_u64(pipe.ctr) == ref["ctr"]).all()


# ------------------------------------------------------------------ f3 token-weighted replay ---
def _fixed_len_stream(rng, n, nkeys, lo=16, hi=5000, spread=1.2):
    keys = _rates_keys(rng, nkeys, n, skew=spread)[:n]
    uk, inv = np.unique(keys, return_inverse=True)
    size_of = rng.integers(lo, hi, size=uk.size).astype(np.uint32)  # one prefix length per key
    return keys, size_of[inv]


@pytest.mark.parametrize("caps,lo,hi", [([24576], 16, 5000), ([1, 100, 3000], 16, 5000),
                                        ([4096, 65536, 2 ** 31], 16, 200),       # 1024-prefix bound
                                        ([5000, 10 ** 6], 1, 3)])
def test_token_replay_parity(P, ctx, caps, lo, hi):
    rng = np.random.default_rng(sum(caps) % 1000 + lo)
    n_rep, R, n = 3, 7, 24000
    keys, plen = _fixed_len_stream(rng, n, int(rng.integers(50, 3000)), lo, hi)
    n = keys.size
    slen = rng.integers(0, 200, size=n).astype(np.uint32)
    dest = tg.random_dest(n_rep, n, R, 5)
    orp = O.Replay(n_rep, R, caps, tokens=True)
    rp = P.Replay(ctx, n_rep, R, caps, tokens=True)
    ctr = torch.zeros((n_rep, len(caps), R, 5), dtype=torch.int64, device=DEV)
    dk, dp, ds, dd = d_u64(keys), d_u32(plen), d_u32(slen), d_u16(dest)
    cut = n // 3
    for a, b in ((0, cut), (cut, n)):  # state persists across calls
        orp.step(keys[a:b], plen[a:b], slen[a:b], dest[:, a:b])
        P.shadow_replay(ctx, rp, dk[a:b].contiguous(), dp[a:b].contiguous(), ds[a:b].contiguous(),
                        dd[:, a:b].contiguous(), ctr)
        ctx.sync()
        assert (h_u64(ctr) == orp.ctr).all()
    ci = caps.index(max(caps))
    for rep in range(n_rep):
        for r in range(R):
            assert (rp.state(rep, r) == orp.state(rep, ci, r)).all()


@pytest.mark.parametrize("caps,lo,hi,nkeys", [([24576], 16, 5000, 400), ([1, 100, 3000], 16, 5000, 2000),
                                              ([4096, 65536, 2 ** 31], 16, 200, 3000)])
def test_token_replay_parity_long_streams(P, ctx, caps, lo, hi, nkeys):
    # streams much longer than the chunks the byte-aware replay splits them into: every chunk
    # after a stream's first rebuilds its starting list by walking back over the stream and
    # the carried-in list, in both calls
    rng = np.random.default_rng(nkeys + lo)
    n_rep, R, n = 2, 2, 80000
    keys, plen = _fixed_len_stream(rng, n, nkeys, lo, hi)
    n = keys.size
    slen = rng.integers(0, 200, size=n).astype(np.uint32)
    dest = tg.random_dest(n_rep, n, R, 8)
    orp = O.Replay(n_rep, R, caps, tokens=True)
    rp = P.Replay(ctx, n_rep, R, caps, tokens=True)
    ctr = torch.zeros((n_rep, len(caps), R, 5), dtype=torch.int64, device=DEV)
    dk, dp, ds, dd = d_u64(keys), d_u32(plen), d_u32(slen), d_u16(dest)
    cut = n // 3
    for a, b in ((0, cut), (cut, n)):
        if a == cut:  # the second call's streams span several chunks at every capacity tested
            assert np.bincount(dest[0, a:b], minlength=R).min() > (16384 if max(caps) > (1 << 17) else 4096)
            # (capacities up to 2^16 tokens use chunks of 1,024 requests, up to 2^17 of 4,096)
        orp.step(keys[a:b], plen[a:b], slen[a:b], dest[:, a:b])
        P.shadow_replay(ctx, rp, dk[a:b].contiguous(), dp[a:b].contiguous(), ds[a:b].contiguous(),
                        dd[:, a:b].contiguous(), ctr)
        ctx.sync()
        assert (h_u64(ctr) == orp.ctr).all()
    ci = caps.index(max(caps))
    for rep in range(n_rep):
        for r in range(R):
            assert (rp.state(rep, r) == orp.state(rep, ci, r)).all()


def test_token_replay_saturating_sums(P, ctx):
    # prefixes near 2^31 tokens: sums past 2^32 saturate and are evicted like any over-capacity run
    caps = [2 ** 31, 2 ** 30]
    keys = np.array([1, 2, 1, 3, 4, 3, 2, 1, 1, 3, 4], np.uint64)
    size = {1: 2 ** 30, 2: 2 ** 31 - 5, 3: 2 ** 31, 4: 2 ** 32 - 1}  # 3 then 4: 3's sum passes 2^32
    plen = np.array([size[int(k)] for k in keys], np.uint32)
    slen = np.zeros(keys.size, np.uint32)
    dest = np.zeros((1, keys.size), np.uint16)
    orp = O.Replay(1, 1, caps, tokens=True)
    orp.step(keys, plen, slen, dest)
    rp = P.Replay(ctx, 1, 1, caps, tokens=True)
    ctr = torch.zeros((1, 2, 1, 5), dtype=torch.int64, device=DEV)
    P.shadow_replay(ctx, rp, d_u64(keys), d_u32(plen), d_u32(slen), d_u16(dest), ctr)
    ctx.sync()
    assert (h_u64(ctr) == orp.ctr).all()
    assert (rp.state(0, 0) == orp.state(0, 0, 0)).all()
    with pytest.raises(P.CacheRouteError):
        P.Replay(ctx, 1, 1, [2 ** 31 + 1], tokens=True)


def test_token_replay_changed_length_is_reported(P, ctx):
    rp = P.Replay(ctx, 1, 2, [10000], tokens=True)
    keys = d_u64(np.array([5, 6, 5], np.uint64))
    plen = d_u32(np.array([100, 200, 150], np.uint32))  # key 5 comes back with another length
    slen = d_u32(np.zeros(3, np.uint32))
    dest = d_u16(np.zeros((1, 3), np.uint16))
    ctr = torch.zeros((1, 1, 2, 5), dtype=torch.int64, device=DEV)
    P.shadow_replay(ctx, rp, keys, plen, slen, dest, ctr)
    with pytest.raises(P.CacheRouteError):
        ctx.sync()
    rp.reset()
    P.shadow_replay(ctx, rp, keys[:2].contiguous(), plen[:2].contiguous(), slen[:2].contiguous(),
                    dest[:, :2].contiguous(), ctr)
    ctx.sync()
    assert rp.state(0, 0).tolist() == [6, 5]


@pytest.mark.parametrize("name,n,nint", [("70b", 40000, 3), ("large", 100000, 2)])
def test_pipeline_parity_token_lru(P, ctx, name, n, nint):
    from paper_2608_19677_gb300.pipeline import Pipeline
    cfg = tg.CONFIGS[name].scaled(n, nint).token_lru()
    if name == "large":  # fewer replicas keep the oracle quick; R, caps and the 1024-prefix bound stay
        import dataclasses
        cfg = dataclasses.replace(cfg, seeds=[0, 1])
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=1024, keep=True)
    pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=1024, overlap=True,
                    lru_tokens=True)
    for t in range(cfg.n_intervals):
        iv = tr.interval(t)
        tok, off = tg.arena_host(tr, iv, 4)
        pipe.interval(t, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), d_u32(iv.slen), iv.g0,
                      plan_next=t + 1 < cfg.n_intervals)
    pipe.sync()
    assert (h_u64(pipe.ctr) == ref["ctr"]).all()


@pytest.mark.parametrize("name,n,nint", [("8b", 6000, 5), ("70b", 30000, 3)])
def test_pipeline_cuda_graph_replay(P, ctx, name, n, nint):
    # a whole step captured once as a CUDA graph (planner and replay streams joined through
    # events) gives the counters of the ordinary step, replay after replay
    from paper_2608_19677_gb300.pipeline import Pipeline
    cfg = tg.CONFIGS[name].scaled(n, nint)
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=1024)
    s = torch.cuda.Stream(DEV)
    with torch.cuda.stream(s):
        gctx = P.Context(0, s)
        ins = []
        for t in range(cfg.n_intervals):
            iv = tr.interval(t)
            tok, off = tg.arena_host(tr, iv, 4)
            ins.append((t, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), d_u32(iv.slen), iv.g0))
        pipe = Pipeline(gctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=1024, overlap=True,
                        max_n=max(int(x[2].shape[0]) for x in ins))

        def step():
            pipe.reset()
            for i, (t, tok, off, pl, sl, g0) in enumerate(ins):
                pipe.interval(t, tok, off, pl, sl, g0, plan_next=i + 1 < len(ins))
            pipe.finish()

        step()
        torch.cuda.synchronize()
        assert (h_u64(pipe.ctr) == ref["ctr"]).all()
        pipe.quiesce()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=s):
            step()
        for _ in range(2):
            pipe.ctr.fill_(-1)
            graph.replay()
            torch.cuda.synchronize()
            assert (h_u64(pipe.ctr) == ref["ctr"]).all()
    gctx.sync()


# ------------------------------------------------------------------ f3 slot-capped placement ---
@pytest.mark.parametrize("R,W,nkeys,total,skew", [(2, 2, 4, 127, 0), (30, 3, 3000, 60000, 1),
                                                  (300, 2, 20000, 700000, 1), (1024, 4, 60000, 300000, 0),
                                                  (3000, 1, 5000, 40000, 1)])
def test_plan_parity_slotcap(P, ctx, R, W, nkeys, total, skew):
    # the capped LPT against the oracle, on the one-CTA build and on the device-wide build
    # (700,000 requests), with and without a skewed starting load (which trims replica counts)
    rng = np.random.default_rng(R + W)
    keys = _rates_keys(rng, nkeys, total)
    n = keys.size
    init = None
    if skew:
        init = rng.integers(0, 50, R).astype(np.uint64)
        init[: max(1, R // 4)] += np.uint64(10 ** 6)
    for num, den in ((5 * n, 4 * R), (n, 20 * R)):
        dl = d_u64(init) if init is not None else None
        got = P.build_plan(ctx, d_u64(keys), P.plan_params(R, W, num, den, "SLOTCAP", init_load=dl)).export()
        ref = O.build_plan(keys, R, W, num, den, variant="SLOTCAP", init_load=init)
        _cmp_plan(got, ref)
        assert np.bincount(got["members"].astype(np.int64), minlength=R).max() <= W


def test_pipeline_parity_slotcap_policy(P, ctx):
    import dataclasses
    from paper_2608_19677_gb300.pipeline import Pipeline
    cfg = dataclasses.replace(tg.CONFIGS["8b"].scaled(8000, 4), policies=["CR", "CR_SLOTCAP", "P2C"], seeds=[0, 1])
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=1024, keep=True)
    pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=1024, overlap=True)
    for t in range(cfg.n_intervals):
        iv = tr.interval(t)
        tok, off = tg.arena_host(tr, iv, 4)
        pipe.interval(t, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), d_u32(iv.slen), iv.g0,
                      plan_next=t + 1 < cfg.n_intervals)
        pipe.wait_last()
        assert (h_u16(pipe.last_dest) == ref["dest"][t]).all()
    pipe.sync()
    assert (h_u64(pipe.ctr) == ref["ctr"]).all()


@pytest.mark.parametrize("B,chwbl", [(1024, False), (1024, True), (1, True)])
def test_pipeline_split_routing_on_sm_partition(P, ctx, B, chwbl):
    # hashing and candidates on the large SM partition, the route resolution on the small one
    # (green contexts): same destinations and counters as the oracle, with the CTA resolution
    # (B = 1024) and the one-warp exact-sequential one (B = 1), with and without bounded-load
    # (ring) replicas
    import dataclasses
    from paper_2608_19677_gb300.pipeline import Pipeline
    try:
        part = P.Partition(0, 16)
    except P.CacheRouteError as e:
        pytest.skip(f"no SM partition on this driver: {e}")
    cfg = tg.CONFIGS["70b"].scaled(40000 if B > 1 else 12000, 4 if B > 1 else 2)
    if chwbl:
        cfg = dataclasses.replace(cfg, policies=["CR", "P2C", "CHWBL"], seeds=[0, 1])
    tr = tg.Trace(cfg)
    ref = OP.run_trace(tr, B=B, keep=True)
    with torch.cuda.stream(part.big):
        pctx = P.Context(0, part.big)
        pipe = Pipeline(pctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=B, overlap=True,
                        resolve_stream=part.small, vnodes=cfg.vnodes)
        for t in range(cfg.n_intervals):
            iv = tr.interval(t)
            tok, off = tg.arena_host(tr, iv, 4)
            pipe.interval(t, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen), d_u32(iv.slen), iv.g0,
                          plan_next=t + 1 < cfg.n_intervals)
            pipe.wait_last()
            assert (h_u16(pipe.last_dest) == ref["dest"][t]).all()
        pipe.sync()
        assert (h_u64(pipe.ctr) == ref["ctr"]).all()
    pipe.close()  # what uses the partition's streams goes before the partition
    pctx.close()
    part.close()


def test_split_route_error_reported_by_sync(P):
    # a bounded-load replica whose load sum has wrapped past 2^64 leaves no destination below
    # cap: the resolution, enqueued on the resolve stream, raises the overflow flag, and the
    # next cr_sync must report it even though the context's own stream finished first
    c = P.Context(0)
    side = torch.cuda.Stream(DEV)
    try:
        R = 2
        ring = P.Ring(c, R, 4, 3)
        P.set_resolve_stream(c, side)
        keys = d_u64(np.arange(1, 65, dtype=np.uint64))
        # loads 2^63 and 2^63 + 2: their sum wraps to 2, so cap = ceil(5 * 3 / 8) = 2 < both
        load = d_u64(np.array([[2 ** 63, 2 ** 63 + 2]], np.uint64))
        P.route_batch(c, [None], ["CHWBL"], [5], R, keys, 0, 64, load, rings=[ring])
        with pytest.raises(P.CacheRouteError) as ei:
            c.sync()
        assert ei.value.code == P.CR_EOVERFLOW
        c.sync()   # reported once, then cleared
        P.set_resolve_stream(c, None)
        ring.close()
    finally:
        c.close()


def test_profile_events_time_each_launch(P):
    # per-launch timing: every timed kind of launch is counted once per call, with a positive duration
    c = P.Context(0)
    try:
        c.profile_enable(64)
        cfg = tg.CONFIGS["70b"].scaled(20000, 1)
        tr = tg.Trace(cfg)
        iv = tr.interval(0)
        tok, off = tg.arena_host(tr, iv, 4)
        keys = P.hash_prefixes(c, torch.from_numpy(tok).to(DEV), d_u64(off), d_u32(iv.plen))
        num, den = tr.qcap(iv.n)
        plan = P.build_plan(c, keys, P.plan_params(cfg.R, cfg.W, num, den, "LPT"))
        load = torch.zeros((2, cfg.R), dtype=torch.int64, device=DEV)
        dest = P.route_batch(c, [plan, None], ["CR", "P2C"], [0, 0], cfg.R, keys, iv.g0, 1024, load)
        rp = P.Replay(c, 2, cfg.R, cfg.caps)
        ctr = torch.zeros((2, 1, cfg.R, 5), dtype=torch.int64, device=DEV)
        P.shadow_replay(c, rp, keys, d_u32(iv.plen), d_u32(iv.slen), dest, ctr)
        c.sync()
        for tag in ("hash", "plan", "route_cand", "route_resolve", "partition", "replay"):
            n, ms = c.profile_read(tag)
            assert n == 1 and ms > 0.0, tag
        c.profile_enable(0)
        assert c.profile_read("replay") == (0, 0.0)
        import ctypes
        n_, ms_ = ctypes.c_uint64(), ctypes.c_double()
        assert P.lib().cr_profile_read(c.handle, 99, ctypes.byref(n_), ctypes.byref(ms_)) == P.CR_EINVAL
        rp.close()
        plan.close()
    finally:
        c.close()


def test_plan_import_routes_like_the_built_plan(P, ctx):
    # a plan exported from the device and installed again (as a host planner's table would
    # be) routes exactly as the plan it came from; bad tables are refused
    rng = np.random.default_rng(21)
    R, W = 64, 8
    keys = _rates_keys(rng, 3000, 60000)
    n = keys.size
    built = P.build_plan(ctx, d_u64(keys), P.plan_params(R, W, 5 * n, 4 * R, "LPT"))
    ex = built.export()
    imp = P.Plan(ctx).load(R, W, ex["adm_key"], ex["adm_cnt"], ex["adm_k"], ex["members"], ex["jobs"], ex["load"])
    got = imp.export()
    for f in ("adm_key", "adm_cnt", "adm_k", "koff", "members", "jobs", "load"):
        assert (got[f] == ex[f]).all(), f
    assert got["n_adm"] == ex["n_adm"] and got["sum_k"] == ex["sum_k"]
    load = torch.zeros((2, R), dtype=torch.int64, device=DEV)
    dk = d_u64(keys)
    d = P.route_batch(ctx, [built, imp], ["CR", "CR"], [3, 3], R, dk, 0, 1024, load)
    ctx.sync()
    h = h_u16(d)
    assert (h[0] == h[1]).all()
    # the oracle agrees with the imported plan's routes
    opl = O.build_plan(keys, R, W, 5 * n, 4 * R)
    od, _ = O.route([opl], ["CR"], [3], R, keys, 0, 1024)
    assert (h[1] == od[0]).all()
    for bad in (dict(adm_k=np.zeros_like(ex["adm_k"])),                       # k = 0
                dict(members=np.full_like(ex["members"], R)),                 # member >= R
                dict(adm_key=np.zeros_like(ex["adm_key"]))):                  # repeated key
        args = dict(adm_key=ex["adm_key"], adm_cnt=ex["adm_cnt"], adm_k=ex["adm_k"], members=ex["members"])
        args.update(bad)
        with pytest.raises(P.CacheRouteError):
            P.Plan(ctx).load(R, W, **args)


def test_replay_state_import_resumes(P, ctx):
    # replay two calls in one simulator set; export every state after the first, import
    # it into a fresh set, and the second call's counters match
    rng = np.random.default_rng(5)
    caps, n_rep, R = [8, 64, 256], 2, 6
    keys = _rates_keys(rng, 2000, 30000)
    n = keys.size
    plen = rng.integers(16, 4000, size=n).astype(np.uint32)
    slen = np.full(n, 64, np.uint32)
    dest = tg.random_dest(n_rep, n, R, 9)
    cut = n // 2
    dk, dp, ds, dd = d_u64(keys), d_u32(plen), d_u32(slen), d_u16(dest)
    a = P.Replay(ctx, n_rep, R, caps)
    ctr_a = torch.zeros((n_rep, len(caps), R, 5), dtype=torch.int64, device=DEV)
    P.shadow_replay(ctx, a, dk[:cut].contiguous(), dp[:cut].contiguous(), ds[:cut].contiguous(),
                    dd[:, :cut].contiguous(), ctr_a)
    ctx.sync()
    b = P.Replay(ctx, n_rep, R, caps)
    for rep in range(n_rep):
        for r in range(R):
            b.set_state(rep, r, a.state(rep, r))
    ctr_a.zero_()
    ctr_b = torch.zeros_like(ctr_a)
    for rp, ctr in ((a, ctr_a), (b, ctr_b)):
        P.shadow_replay(ctx, rp, dk[cut:].contiguous(), dp[cut:].contiguous(), ds[cut:].contiguous(),
                        dd[:, cut:].contiguous(), ctr)
    ctx.sync()
    assert (h_u64(ctr_a) == h_u64(ctr_b)).all()
    with pytest.raises(P.CacheRouteError):
        b.set_state(0, 0, np.array([1, 2, 1], np.uint64))     # repeated key
    with pytest.raises(P.CacheRouteError):
        b.set_state(0, R, np.array([1], np.uint64))            # no such destination
    a.close()
    b.close()


def test_debug_build_runs_the_smoke_check_clean():
    # the bounds-checking build gives the oracle's results and raises no flag on a small
    # pass of the whole path (run in a child process that loads the debug library)
    import os
    import subprocess
    import sys
    from paper_2608_19677_gb300 import buildlib
    buildlib.build(debug=True)
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, CR_DEBUG_LIB="1")
    code = ("import paper_2608_19677_gb300 as P, __graft_entry__ as g; "
            "assert P.LIB_PATH.endswith('libcacheroute_debug.so'); g.smoke()")
    r = subprocess.run([sys.executable, "-c", code], cwd=root, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    assert "smoke ok" in r.stdout


def test_replay_partition_then_simulate_equals_shadow_replay(P, ctx):
    # the two-call form (partition on one stream, simulation on another, ordered by an
    # event) gives the same counters and states as cr_shadow_replay, over two calls; an
    # input partitioned for another replay shape is refused
    rng = np.random.default_rng(17)
    caps, n_rep, R = [16, 64], 3, 9
    keys = _rates_keys(rng, 800, 24000)
    n = keys.size
    plen = rng.integers(16, 3000, size=n).astype(np.uint32)
    slen = np.full(n, 64, np.uint32)
    dest = tg.random_dest(n_rep, n, R, 4)
    dk, dp, ds, dd = d_u64(keys), d_u32(plen), d_u32(slen), d_u16(dest)
    a = P.Replay(ctx, n_rep, R, caps)
    b = P.Replay(ctx, n_rep, R, caps)
    ctr_a = torch.zeros((n_rep, len(caps), R, 5), dtype=torch.int64, device=DEV)
    ctr_b = torch.zeros_like(ctr_a)
    side = torch.cuda.Stream(DEV)
    pctx = P.Context(0, side)
    inp = P.ReplayInput(pctx)
    cut = n // 2
    for lo, hi in ((0, cut), (cut, n)):
        args = (dk[lo:hi].contiguous(), dp[lo:hi].contiguous(), ds[lo:hi].contiguous(), dd[:, lo:hi].contiguous())
        P.shadow_replay(ctx, a, *args, ctr_a)
        side.wait_stream(torch.cuda.current_stream(DEV))
        P.replay_partition(pctx, b, *args, inp)
        ev = torch.cuda.Event()
        ev.record(side)
        torch.cuda.current_stream(DEV).wait_event(ev)
        P.replay_simulate(ctx, b, inp, ctr_b)
        ctx.sync()
        pctx.sync()
    assert (h_u64(ctr_a) == h_u64(ctr_b)).all()
    for rep in range(n_rep):
        for r in range(R):
            assert (a.state(rep, r) == b.state(rep, r)).all()
    other = P.Replay(ctx, n_rep, R + 1, caps)
    with pytest.raises(P.CacheRouteError):
        P.replay_simulate(ctx, other, inp, torch.zeros((n_rep, len(caps), R + 1, 5), dtype=torch.int64, device=DEV))
    inp.close()
    pctx.close()
