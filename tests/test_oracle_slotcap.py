"""Pins for the oracle's slot-capped placement variant (CPU only).

Byte-aware placement (a per-destination budget, this library's reading of the
paper's byte budgets): LPT as in Algorithm 1, but a destination holds at most
W replicas; a key goes to the k smallest (L, r) among destinations with a free
slot, with k = min(k_b, such destinations).  Pins: the cap holds in every
plan; when it cannot bind (W at least the number of admitted keys) the plan is
the plain LPT plan, member for member; a hand-worked plan where the cap moves
a key; a hand-worked plan where it trims a key's replica count; admission and
job conservation are unchanged.
"""
import numpy as np
import pytest

import oracle as O


def _keys(counts):
    return np.repeat(np.arange(1, len(counts) + 1, dtype=np.uint64) * np.uint64(0x9E3779B97F4A7C15),
                     counts)


@pytest.mark.parametrize("seed", range(6))
def test_cap_holds_and_jobs_are_conserved(seed):
    rng = np.random.default_rng(seed)
    R = int(rng.integers(2, 40))
    W = int(rng.integers(1, 6))
    keys = (rng.zipf(1.3, 20000) % 3000).astype(np.uint64) * np.uint64(0x9E3779B97F4A7C15)
    num, den = keys.size, int(rng.integers(1, 6)) * R
    init = rng.integers(0, 500, R).astype(np.uint64) if seed % 2 else None
    pc = O.build_plan(keys, R, W, num, den, variant="SLOTCAP", init_load=init)
    pl = O.build_plan(keys, R, W, num, den, variant="LPT", init_load=init)
    assert pc.n_adm == pl.n_adm and (pc.adm_key == pl.adm_key).all()    # admission unchanged
    assert np.bincount(pc.members.astype(np.int64), minlength=R).max() <= W
    assert (pc.adm_k >= 1).all() and (pc.adm_k <= pl.adm_k).all()
    assert pc.sum_k == int(pc.adm_k.sum()) == pc.members.size
    for e in range(pc.n_adm):
        ms = pc.members[pc.koff[e]:pc.koff[e + 1]]
        assert len(set(ms.tolist())) == ms.size == pc.adm_k[e]            # distinct destinations
        assert int(pc.jobs[pc.koff[e]:pc.koff[e + 1]].sum()) == int(pc.adm_cnt[e])
    base = init.astype(np.int64) if init is not None else np.full(R, pc.cold // R, np.int64)
    assert (pc.load.astype(np.int64) - base).sum() == int(pc.adm_cnt.sum())


@pytest.mark.parametrize("seed", range(4))
def test_no_binding_cap_is_plain_lpt(seed):
    rng = np.random.default_rng(10 + seed)
    R = int(rng.integers(2, 30))
    keys = (rng.zipf(1.2, 8000) % 500).astype(np.uint64) * np.uint64(0x9E3779B97F4A7C15)
    W = 600  # at least the number of admitted keys: the cap never binds
    a = O.build_plan(keys, R, W, keys.size, 3 * R, variant="SLOTCAP")
    b = O.build_plan(keys, R, W, keys.size, 3 * R, variant="LPT")
    assert (a.members == b.members).all() and (a.koff == b.koff).all() and (a.load == b.load).all()


def test_hand_plan_cap_moves_a_key():
    # R = 2, W = 2 (C = 4), q_cap = 1000 so every k_b = 1, no cold tail.  Rates 100, 10, 9, 8.
    # LPT: 100 -> d0; 10 -> d1; 9 -> d1 (L1 10 < 100); 8 -> d1 (19 < 100): d1 holds 3 keys.
    # Capped: d1 is full after 10 and 9, so 8 goes to d0.
    keys = _keys([100, 10, 9, 8])
    lpt = O.build_plan(keys, 2, 2, 1000, 1, variant="LPT")
    cap = O.build_plan(keys, 2, 2, 1000, 1, variant="SLOTCAP")
    assert lpt.members.tolist() == [0, 1, 1, 1]
    assert cap.members.tolist() == [0, 1, 1, 0]
    assert cap.load.tolist() == [108, 19]


def test_hand_plan_cap_trims_replicas():
    # R = 3, W = 2 (C = 6), q_cap = 5: three keys of 10 requests, k_b = 2 each; d0 starts
    # with load 1000.  Keys 1 and 2 take d1 and d2 (filling them); key 3 finds only d0 with
    # a free slot and gets one replica carrying all 10 requests.
    keys = _keys([10, 10, 10])
    init = np.array([1000, 0, 0], np.uint64)
    cap = O.build_plan(keys, 3, 2, 5, 1, variant="SLOTCAP", init_load=init)
    assert cap.adm_k.tolist() == [2, 2, 1]
    assert cap.koff.tolist() == [0, 2, 4, 5]
    assert sorted(cap.members[:2].tolist()) == [1, 2] and sorted(cap.members[2:4].tolist()) == [1, 2]
    assert cap.members[4] == 0 and cap.jobs[4] == 10 and cap.sum_k == 5
    assert cap.load.tolist() == [1010, 10, 10]
