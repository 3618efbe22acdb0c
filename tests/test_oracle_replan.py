"""Pins for the replanning-under-drift pieces of the oracle (CPU only).

Cache churn is 1 - Jaccard of two consecutive assignment sets ((key,
destination) pairs of T); count churn is the share of keys whose k_b changes
(supplement "Replanning Under Drift", replan table; sec. 5 "Rate drift and
remapping").  The pins are hand-built plans with hand-counted answers, the
Jaccard index of key x destination incidence matrices (numpy, no sets),
identity and symmetry, and the structural case the paper points out: every
key keeps k_b = 1 but moves to another destination (cache churn 1, count churn 0).
The drift generator is pinned by its defining distribution: log-share steps
are N(0, sigma^2) and interval 0 keeps the primary shares.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle as O
import tracegen as tg


def _plan(R, table, hist=None, qcap=(1, 1), variant="LPT"):
    """An oracle Plan holding an admitted table {key: [members]} (admission order = dict order)
    and a histogram {key: lambda} (default: lambda = 1 for every admitted key)."""
    keys = list(table)
    ks = [len(table[k]) for k in keys]
    koff = np.concatenate([[0], np.cumsum(ks)]).astype(np.uint32)
    mem = np.array([d for k in keys for d in table[k]], np.uint16)
    pl = O.Plan(R, 1, len(keys), len(keys), int(sum(ks)), 0, np.array(keys, np.uint64),
                np.ones(len(keys), np.uint64), np.array(ks, np.uint32), koff, mem,
                np.zeros(mem.size, np.uint64), np.zeros(R, np.uint64))
    hist = hist if hist is not None else {k: 1 for k in keys}
    pl.hist_key = np.array(list(hist), np.uint64)
    pl.hist_cnt = np.array(list(hist.values()), np.uint64)
    pl.qcap, pl.variant = qcap, variant
    return pl


def _eq1(lam, num, den, R):
    # k_b = max(1, ceil(lambda / q_cap)) clamped to R, q_cap = num / den, by exact fractions
    return min(R, max(1, -(-Fraction(lam) // Fraction(num, den))))


def test_hand_built_plans():
    a = _plan(6, {10: [0], 11: [1, 2], 12: [3], 13: [4, 5, 0]},
              hist={10: 5, 11: 9, 12: 2, 13: 14, 16: 1}, qcap=(4, 1))
    b = _plan(6, {11: [2, 1], 12: [4], 13: [4, 5], 14: [3]},
              hist={11: 9, 12: 6, 13: 10, 14: 3, 15: 1}, qcap=(5, 1))
    d = O.plan_diff(a, b)
    # pairs a: (10,0) (11,1) (11,2) (12,3) (13,4) (13,5) (13,0) = 7
    # pairs b: (11,2) (11,1) (12,4) (13,4) (13,5) (14,3) = 6; common: (11,1) (11,2) (13,4) (13,5) = 4
    # Eq. 1 under a (q_cap 4): 10:2 11:3 12:1 13:4 16:1, absent 14,15: 1
    # Eq. 1 under b (q_cap 5): 11:2 12:2 13:2 14:1 15:1, absent 10,16: 1 -> 10,11,12,13 change
    assert d == dict(keys_a=4, keys_b=4, keys_common=3, pairs_a=7, pairs_b=6, pairs_common=4,
                     adm_k_changed=3,      # 10 (1 -> 0), 13 (3 -> 2), 14 (0 -> 1)
                     adm_set_changed=4,    # 10, 12, 13, 14 (11 keeps {1, 2} in another order)
                     hist_keys=7, hist_kb_changed=4)
    cache, count = O.churn(d)
    assert cache == 1 - Fraction(4, 9) and count == Fraction(4, 7)


def _random_plan(rng, R, nkeys, universe, kmax):
    keys = rng.choice(universe, size=nkeys, replace=False)
    hk = rng.choice(universe, size=int(rng.integers(nkeys, universe + 1)), replace=False)
    hist = {int(k): int(rng.integers(1, 60)) for k in np.union1d(keys, hk)}
    q = (int(rng.integers(1, 40)), int(rng.integers(1, 5)))
    return _plan(R, {int(k): [int(x) for x in rng.choice(R, size=int(rng.integers(1, kmax + 1)),
                                                          replace=False)] for k in keys},
                 hist=hist, qcap=q, variant="NOREPL" if rng.random() < 0.2 else "LPT")


@pytest.mark.parametrize("seed", range(8))
def test_against_incidence_matrices(seed):
    rng = np.random.default_rng(seed)
    R = int(rng.integers(1, 40))
    a = _random_plan(rng, R, int(rng.integers(0, 60)), 90, min(R, 5))
    b = _random_plan(rng, R, int(rng.integers(0, 60)), 90, min(R, 5))
    A = np.zeros((90, R), bool)
    B = np.zeros((90, R), bool)
    for M, p in ((A, a), (B, b)):
        for e in range(p.n_adm):
            M[int(p.adm_key[e]), p.members[p.koff[e]:p.koff[e + 1]].astype(np.int64)] = True
    d = O.plan_diff(a, b)
    assert d["pairs_common"] == int((A & B).sum())
    assert d["pairs_a"] + d["pairs_b"] - d["pairs_common"] == int((A | B).sum())
    ka, kb = A.sum(1), B.sum(1)
    either = (ka > 0) | (kb > 0)
    assert d["adm_k_changed"] == int((ka != kb)[either].sum())
    assert d["adm_set_changed"] == int((A != B).any(1)[either].sum())
    # count churn over the union of histograms, lambda = 0 where a key is missing
    lam = np.zeros((2, 90), np.int64)
    for i, p in enumerate((a, b)):
        lam[i, p.hist_key.astype(np.int64)] = p.hist_cnt.astype(np.int64)
    seen = (lam > 0).any(0)
    kbs = [[1 if p.variant == "NOREPL" else _eq1(int(x), p.qcap[0], p.qcap[1], R) for x in lam[i]]
           for i, p in enumerate((a, b))]
    assert d["hist_keys"] == int(seen.sum())
    assert d["hist_kb_changed"] == int(sum(1 for u in range(90) if seen[u] and kbs[0][u] != kbs[1][u]))
    cache, _ = O.churn(d)
    if (A | B).any():
        assert cache == 1 - Fraction(int((A & B).sum()), int((A | B).sum()))
    rev = O.plan_diff(b, a)
    assert (rev["pairs_a"], rev["keys_a"]) == (d["pairs_b"], d["keys_b"])
    sym = ("keys_common", "pairs_common", "adm_k_changed", "adm_set_changed", "hist_keys", "hist_kb_changed")
    assert {k: rev[k] for k in sym} == {k: d[k] for k in sym}


def test_identity_and_moved_keys():
    a = _plan(5, {1: [0], 2: [1], 3: [2], 4: [3]})
    assert O.churn(O.plan_diff(a, a)) == (0, 0)
    b = _plan(5, {1: [1], 2: [2], 3: [3], 4: [4]})  # same k_b everywhere, every key moved
    assert O.churn(O.plan_diff(a, b)) == (1, 0)
    e = _plan(5, {})
    assert O.churn(O.plan_diff(e, e)) == (0, 0)


def test_single_copy_plans_have_no_count_churn():
    a = _plan(8, {1: [0]}, hist={1: 100, 2: 3}, qcap=(10, 1), variant="NOREPL")
    b = _plan(8, {2: [1]}, hist={1: 2, 2: 90, 3: 7}, qcap=(10, 1), variant="NOREPL")
    d = O.plan_diff(a, b)
    assert d["hist_keys"] == 3 and d["hist_kb_changed"] == 0


def test_real_plans_same_interval_different_placement():
    # two plans of the same interval built with different RANDOM seeds admit the same
    # keys with the same k_b: count churn 0, cache churn from placement only
    rng = np.random.default_rng(3)
    keys = (rng.zipf(1.3, 20000) % 3000).astype(np.uint64) * np.uint64(0x9E3779B97F4A7C15)
    a = O.build_plan(keys, 16, 8, keys.size, 4 * 16, variant="RANDOM", seed=1)
    b = O.build_plan(keys, 16, 8, keys.size, 4 * 16, variant="RANDOM", seed=2)
    d = O.plan_diff(a, b)
    assert d["keys_common"] == d["keys_a"] == d["keys_b"] and d["adm_k_changed"] == 0
    assert d["hist_kb_changed"] == 0 and d["hist_keys"] == np.unique(keys).size
    assert d["pairs_a"] == a.sum_k and 0 < d["pairs_common"] < d["pairs_a"]


def test_drift_generator_is_a_lognormal_walk():
    cfg = tg.CONFIGS["drift"]
    tr = tg.Trace(cfg)
    assert np.array_equal(tr.shares(0), tr.key_p)
    prev = np.log(tr.shares(0))
    for t in range(1, cfg.n_intervals):
        cur = np.log(tr.shares(t))
        step = cur - prev
        step -= step.mean()          # renormalisation shifts every log-share by one constant
        assert abs(step.std() - cfg.drift) < 0.01
        assert abs(np.mean(step ** 3)) < 0.01 * cfg.drift ** 3 * 10  # symmetric
        prev = cur
    assert all(abs(tr.shares(t).sum() - 1) < 1e-12 for t in range(cfg.n_intervals))


def test_gamma_arrivals_have_the_configured_cv():
    cfg = tg.CONFIGS["70b-gamma"]
    tr = tg.Trace(cfg)
    t = tr.arrival_times()
    gaps = np.diff(t)
    assert abs(gaps.std() / gaps.mean() - cfg.arrival_cv) < 0.02
    assert t[0] >= 0 and t[-1] < cfg.n_intervals * cfg.interval_s
    assert tr.counts.sum() == cfg.n_requests
    assert np.array_equal(tr.counts, np.histogram(t, bins=cfg.n_intervals,
                                                  range=(0, cfg.n_intervals * cfg.interval_s))[0])
    # the Poisson configuration is unchanged by the option
    assert tg.CONFIGS["70b"].arrival_cv is None
