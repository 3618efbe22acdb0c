"""Pins for the oracle's dispatch and shadow replay (CPU only).

Dispatch follows Fig. 1 and sec. 3.1 (least-loaded member of T(b), otherwise
power-of-two choices); the replay is this library's whole-prefix LRU reading
of the shadow-replay gate (sec. 3.2, 5.3).  Pins use numpy's Philox (an independent
implementation) to hand-step P2C, Lamping and Veach's monotonicity property of
jump hashing, Mattson's stack-distance characterisation of LRU computed by
brute force, and hand-worked traces.
"""
import json
import os

import numpy as np
import pytest

import oracle as O
import tracegen as tg

M64 = (1 << 64) - 1


def _np_philox(ctr, key):
    # numpy's Philox emits philox(c + 1) for state c (256-bit counter): start one below.
    c = sum(int(w) << (64 * i) for i, w in enumerate(ctr))
    c = (c - 1) % (1 << 256)
    words = [(c >> (64 * i)) & M64 for i in range(4)]
    bg = np.random.Philox(key=np.array(key, dtype=np.uint64),
                         counter=np.array(words, dtype=np.uint64))
    return [int(x) for x in bg.random_raw(4)]


def _hand_p2c(seed, policy_id, g, R, load):
    u = _np_philox([g, 0, 0, 0], [seed, policy_id])
    d1 = (u[0] * R) >> 64
    d2 = (d1 + 1 + ((u[1] * (R - 1)) >> 64)) % R
    return d1 if load[d1] <= load[d2] else d2


def _keys(n, nk, seed=0):
    rng = np.random.default_rng(seed)
    w = 1.0 / np.arange(1, nk + 1)
    kid = rng.choice(nk, size=n, p=w / w.sum())
    return (kid.astype(np.uint64) * np.uint64(0x9E3779B97F4A7C15)) ^ np.uint64(12345)


@pytest.mark.parametrize("R", [1, 2, 7, 30])
def test_p2c_sequential_matches_hand_stepped(R):
    keys = _keys(400, 50)
    dest, load = O.route([None], ["P2C"], [11], R, keys, g0=1000, B=1)
    L = [0] * R
    for i in range(keys.size):
        d = _hand_p2c(11, O.POLICY["P2C"], 1000 + i, R, L)
        assert dest[0, i] == d
        L[d] += 1
    assert load[0].tolist() == L


def test_batch_snapshot_semantics():
    keys = _keys(300, 40)
    R = 9
    # one batch: everybody sees the all-zero snapshot and takes its first choice
    dest, load = O.route([None], ["P2C"], [3], R, keys, g0=0, B=10_000)
    for i in range(keys.size):
        u = _np_philox([i, 0, 0, 0], [3, O.POLICY["P2C"]])
        assert dest[0, i] == (u[0] * R) >> 64
    # batches of 16: the snapshot changes only at batch boundaries
    dest, load = O.route([None], ["P2C"], [3], R, keys, g0=0, B=16)
    L = [0] * R
    for b0 in range(0, keys.size, 16):
        snap = list(L)
        for i in range(b0, min(keys.size, b0 + 16)):
            d = _hand_p2c(3, O.POLICY["P2C"], i, R, snap)
            assert dest[0, i] == d
            L[d] += 1
    assert load[0].tolist() == L


def test_conservation_rr_and_hash():
    keys = _keys(5000, 300, 1)
    R = 13
    dest, load = O.route([None, None, None], ["RR", "HASH", "P2C"], [5, 5, 5], R, keys, g0=77, B=64)
    for rp in range(3):
        assert int(load[rp].sum()) == keys.size
        assert np.bincount(dest[rp], minlength=R).tolist() == load[rp].tolist()
    rr = np.bincount(dest[0], minlength=R)
    assert rr.max() - rr.min() <= 1
    assert dest[0, 0] == (77 + 5) % R
    # sticky: every request of a key goes to one destination
    for k in np.unique(keys)[:100]:
        assert len(set(dest[1, keys == k].tolist())) == 1
    # the HASH choice depends on the key only, not on load or batch
    d2, _ = O.route([None], ["HASH"], [5], R, keys, g0=0, B=1, load=np.full((1, R), 99, np.uint64))
    assert (d2[0] == dest[1]).all()


def test_jump_hash_consistency_and_balance():
    rng = np.random.default_rng(9)
    ks = [int(x) for x in rng.integers(0, 1 << 63, size=3000)]
    for k in ks[:500]:
        assert O.jump_hash(k, 1) == 0
        prev = O.jump_hash(k, 1)
        for R in range(2, 40):
            cur = O.jump_hash(k, R)
            # Lamping and Veach: growing R moves a key only onto the new bucket
            assert cur == prev or cur == R - 1
            prev = cur
    R = 16
    c = np.bincount([O.jump_hash(k, R) for k in ks], minlength=R)
    exp = len(ks) / R
    assert float(((c - exp) ** 2 / exp).sum()) < 45.0   # 15 dof


def _plan_for(keys, R, W, variant="LPT", seed=0):
    n = keys.size
    return O.build_plan(keys, R, W, 5 * n, 4 * R, variant=variant, seed=seed)


@pytest.mark.parametrize("B", [1, 32, 1000])
def test_cacheroute_dispatch(B):
    keys = _keys(3000, 200, 2)
    R = 6
    pl = O.build_plan(keys, R, 4, keys.size, 12 * R)   # tight q_cap: several k_b > 1
    assert (pl.adm_k > 1).any()
    tab = pl.table()
    dest, load = O.route([pl], ["CR"], [4], R, keys, g0=0, B=B)
    L = [0] * R
    for b0 in range(0, keys.size, B):
        snap = list(L)
        for i in range(b0, min(keys.size, b0 + B)):
            k = int(keys[i])
            if k in tab:
                mem = tab[k]
                # least-loaded member of T(b); ties keep the earlier member
                want = min(mem, key=lambda m: (snap[m], mem.index(m)))
            else:
                want = _hand_p2c(4, O.POLICY["CR"], i, R, snap)
            assert dest[0, i] == want
            L[want] += 1
    assert load[0].tolist() == L


def test_cacheroute_k1_goes_to_its_single_member():
    keys = _keys(4000, 100, 3)
    R = 4
    pl = _plan_for(keys, R, 5)
    assert (pl.adm_k == 1).all()
    tab = pl.table()
    dest, _ = O.route([pl], ["CR"], [0], R, keys, g0=0, B=256)
    for i in range(keys.size):
        k = int(keys[i])
        if k in tab:
            assert dest[0, i] == tab[k][0]


# -------------------------------------------------------------------------
# replay
# -------------------------------------------------------------------------
def _replay(stream, caps, plen=10, slen=2, R=1, dest=None):
    n = len(stream)
    rp = O.Replay(1, R, caps)
    d = np.zeros((1, n), np.uint16) if dest is None else dest
    rp.step(np.asarray(stream, np.uint64), np.full(n, plen, np.uint32), np.full(n, slen, np.uint32), d)
    return rp


def test_lru_hand_trace(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "lru_hand_trace.json")))
    caps = [int(c) for c in g["expect"]]
    rp = _replay(g["stream"], caps, g["plen"], g["slen"])
    for ci, c in enumerate(caps):
        e = g["expect"][str(c)]
        got = rp.ctr[0, ci, 0]
        assert got.tolist() == [len(g["stream"]), e["hits"], e["hit_tokens"], e["prompt_tokens"],
                                e["prefill_tokens"]]
        assert rp.state(0, ci, 0).tolist() == e["final"]


def _stack_distances(stream):
    """Mattson stack distance by brute force: 1 + distinct keys since the last use."""
    out = []
    for t, x in enumerate(stream):
        prev = None
        for u in range(t - 1, -1, -1):
            if stream[u] == x:
                prev = u
                break
        out.append(None if prev is None else 1 + len(set(stream[prev + 1:t])))
    return out


@pytest.mark.parametrize("seed", range(5))
def test_lru_equals_stack_distance_rule(seed):
    rng = np.random.default_rng(seed)
    nk = int(rng.integers(2, 40))
    stream = rng.zipf(1.3, size=400) % nk
    caps = [1, 2, 3, 5, 8, 16, 64]
    rp = _replay(stream.tolist(), caps)
    sd = _stack_distances(stream.tolist())
    hits = [rp.ctr[0, ci, 0, 1] for ci in range(len(caps))]
    for ci, c in enumerate(caps):
        assert hits[ci] == sum(1 for d in sd if d is not None and d <= c)
    assert all(a <= b for a, b in zip(hits, hits[1:]))   # inclusion
    # capacity >= distinct keys: hits = requests - distinct keys
    assert hits[-1] == len(stream) - len(set(stream.tolist()))
    # capacity 1: a hit exactly when the previous request had the same key
    assert hits[0] == int((stream[1:] == stream[:-1]).sum())


def test_replay_counters_destinations_and_persistence():
    rng = np.random.default_rng(11)
    n, R, n_rep = 3000, 5, 3
    keys = _keys(n, 80, 4)
    plen = rng.integers(16, 3000, size=n).astype(np.uint32)
    slen = np.full(n, 64, np.uint32)
    dest = tg.random_dest(n_rep, n, R, 5)
    caps = [4, 32]
    one = O.Replay(n_rep, R, caps)
    one.step(keys, plen, slen, dest)
    two = O.Replay(n_rep, R, caps)
    two.step(keys[:1234], plen[:1234], slen[:1234], dest[:, :1234])
    two.step(keys[1234:], plen[1234:], slen[1234:], dest[:, 1234:])
    assert (one.ctr == two.ctr).all()
    c = one.ctr
    assert (c[..., 4] == c[..., 3] - c[..., 2]).all()          # prefill = prompt - hit tokens
    for rp in range(n_rep):
        for ci in range(len(caps)):
            assert int(c[rp, ci, :, 0].sum()) == n
            assert int(c[rp, ci, :, 3].sum()) == int(plen.sum() + slen.sum())
            for r in range(R):
                sel = dest[rp] == r
                assert c[rp, ci, r, 0] == sel.sum()
                sd = _stack_distances(keys[sel].tolist())
                assert c[rp, ci, r, 1] == sum(1 for d in sd if d is not None and d <= caps[ci])
                hit_tok = sum(int(p) for p, d in zip(plen[sel], sd) if d is not None and d <= caps[ci])
                assert c[rp, ci, r, 2] == hit_tok


def _jump_hash_float(keys: np.ndarray, R: np.ndarray) -> np.ndarray:
    """Lamping and Veach's published jump consistent hash, restated with its
    floating-point bucket jump j = (b + 1) * (2^31 / ((key >> 33) + 1)) in IEEE
    doubles (numpy, vectorised over keys): an independent statement of the
    linear congruential step and of the jump that the oracle evaluates exactly
    in integers."""
    k = keys.astype(np.uint64).copy()
    R = R.astype(np.int64)
    b = np.full(k.shape, -1, np.int64)
    j = np.zeros(k.shape, np.int64)
    live = j < R
    with np.errstate(over="ignore"):
        while live.any():
            b[live] = j[live]
            k[live] = k[live] * np.uint64(2862933555777941757) + np.uint64(1)
            step = float(1 << 31) / ((k[live] >> np.uint64(33)).astype(np.float64) + 1.0)
            j[live] = ((b[live] + 1).astype(np.float64) * step).astype(np.int64)
            live = j < R
    return b


def test_jump_hash_matches_the_published_floating_point_algorithm():
    # 100,000 keys at a random bucket count each, plus 200 keys at every bucket count
    # 1..1024: the oracle's integer jump must pick the same bucket as the published
    # algorithm (a wrong multiplier, increment or shift moves most keys)
    rng = np.random.default_rng(2014)
    keys = rng.integers(0, 1 << 63, size=100000, dtype=np.int64).astype(np.uint64) * np.uint64(2) + \
        rng.integers(0, 2, size=100000).astype(np.uint64)
    R = rng.integers(1, 1025, size=keys.size)
    want = _jump_hash_float(keys, R)
    got = np.array([O.jump_hash(int(k), int(r)) for k, r in zip(keys, R)], np.int64)
    assert (got == want).all(), int((got != want).sum())
    few = keys[:200]
    allR = np.arange(1, 1025)
    kk = np.repeat(few, allR.size)
    rr = np.tile(allR, few.size)
    want = _jump_hash_float(kk, rr)
    got = np.array([O.jump_hash(int(k), int(r)) for k, r in zip(kk, rr)], np.int64)
    assert (got == want).all(), int((got != want).sum())
    # a planted change of the multiplier is caught by the same comparison
    def planted(k, R):
        b, j = -1, 0
        while j < R:
            b = j
            k = (k * 2862933555777941759 + 1) & ((1 << 64) - 1)
            j = int((b + 1) * (float(1 << 31) / float((k >> 33) + 1)))
        return b
    bad = np.array([planted(int(k), int(r)) for k, r in zip(keys[:2000], R[:2000])])
    assert (bad != _jump_hash_float(keys[:2000], R[:2000])).mean() > 0.5
