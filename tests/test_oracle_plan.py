"""Pins for the oracle's plan (Eq. 1 and Algorithm 1, sec. 3.1), CPU only."""
import collections
import fractions
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle as O


def _keys_from_rates(rates, seed=0):
    ks = np.concatenate([np.full(c, k, np.uint64) for k, c in rates.items()])
    np.random.default_rng(seed).shuffle(ks)
    return ks


def test_histogram_matches_counter():
    rng = np.random.default_rng(3)
    keys = rng.integers(0, 50, size=2000).astype(np.uint64) * np.uint64(0x9E3779B97F4A7C15)
    uk, ct = O.histogram(keys)
    ref = collections.Counter(keys.tolist())
    assert sorted(ref) == uk.tolist()
    assert [ref[k] for k in uk.tolist()] == ct.tolist()
    assert int(ct.sum()) == keys.size
    assert O.histogram(np.zeros(0, np.uint64))[0].size == 0


def test_hand_worked_plan(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "plan_hand_example.json")))
    rates = {int(k): v for k, v in g["rates"].items()}
    pl = O.build_plan(_keys_from_rates(rates), g["R"], g["W"], g["qcap_num"], g["qcap_den"])
    e = g["expect"]
    assert pl.n_adm == e["n_adm"] and pl.U == e["U"] and pl.cold == e["cold"]
    assert pl.adm_key.tolist() == e["adm_key"]
    assert pl.adm_k.tolist() == e["adm_k"]
    assert pl.koff.tolist() == e["koff"]
    assert pl.members.tolist() == e["members"]
    assert pl.jobs.tolist() == e["jobs"]
    assert pl.load.tolist() == e["load"]


def test_eq1_against_exact_fractions():
    rng = np.random.default_rng(4)
    for _ in range(3000):
        lam = int(rng.integers(1, 1 << 31))
        num = int(rng.integers(1, 1 << 40))
        den = int(rng.integers(1, 1 << 31))
        R = int(rng.integers(1, 2000))
        q = fractions.Fraction(num, den)
        ref = min(R, max(1, math.ceil(fractions.Fraction(lam) / q)))
        assert O.kb(lam, num, den, R) == ref
    # exact boundary: lambda == q_cap gives one destination, one more gives two
    assert O.kb(12, 12, 1, 8) == 1 and O.kb(13, 12, 1, 8) == 2


def _random_rates(rng, nkeys, total):
    w = rng.pareto(1.2, size=nkeys) + 1e-3
    c = np.maximum(1, np.round(w / w.sum() * total)).astype(np.int64)
    return {int(k) * 7919 + 11: int(v) for k, v in enumerate(c)}


def _brute_admission(rates, R, W, num, den, norepl=False):
    order = sorted(rates.items(), key=lambda kv: (-kv[1], kv[0]))
    C, s, adm = R * W, 0, []
    for k, lam in order:
        kb = 1 if norepl else min(R, max(1, math.ceil(fractions.Fraction(lam * den, num))))
        if s + kb > C:
            break
        s += kb
        adm.append((k, lam, kb))
    return adm


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("variant", ["LPT", "NOREPL", "RANDOM"])
def test_admission_and_placement_invariants(seed, variant):
    rng = np.random.default_rng(100 + seed)
    R = int(rng.integers(1, 24))
    W = int(rng.integers(1, 6))
    rates = _random_rates(rng, int(rng.integers(1, 120)), int(rng.integers(50, 5000)))
    N = sum(rates.values())
    num, den = 5 * N, 4 * R
    if seed % 2:
        num, den = N, 7 * R          # a tighter q_cap forces replication
    pl = O.build_plan(_keys_from_rates(rates, seed), R, W, num, den, variant=variant, seed=seed)
    adm = _brute_admission(rates, R, W, num, den, norepl=(variant == "NOREPL"))
    # admission: the longest (lambda desc, key asc) prefix with sum k_b <= C
    assert pl.adm_key.tolist() == [a[0] for a in adm]
    assert pl.adm_cnt.tolist() == [a[1] for a in adm]
    assert pl.adm_k.tolist() == [a[2] for a in adm]
    assert pl.sum_k == sum(a[2] for a in adm) <= R * W
    assert pl.U == len(rates)
    cold = N - sum(a[1] for a in adm)
    assert pl.cold == cold
    L = [cold // R] * R
    qcap = fractions.Fraction(num, den)
    for a, (k, lam, kb) in enumerate(adm):
        mem = pl.members[pl.koff[a]:pl.koff[a + 1]].tolist()
        jobs = pl.jobs[pl.koff[a]:pl.koff[a + 1]].tolist()
        assert len(mem) == kb and len(set(mem)) == kb and all(0 <= m < R for m in mem)
        # conservation and near-equal split, larger jobs first
        assert sum(jobs) == lam and max(jobs) - min(jobs) <= 1 and jobs == sorted(jobs, reverse=True)
        if variant == "LPT" and kb < R:
            # the expected load per assignment is at most q_cap (sec. 3.1, after Eq. 1)
            assert all(j <= math.ceil(qcap) for j in jobs)
        if variant != "RANDOM":
            # members are the kb smallest (L, r), in that order
            want = sorted(range(R), key=lambda r: (L[r], r))[:kb]
            assert mem == want
        for m, j in zip(mem, jobs):
            L[m] += j
    assert pl.load.tolist() == L


def test_all_kb_one_when_hottest_below_qcap():
    # sec. 3.2: max lambda < q_cap implies k_b = 1 for every key, and Algorithm 1
    # reduces to top-rate admission plus single-copy placement.
    rng = np.random.default_rng(7)
    rates = {i: int(rng.integers(1, 40)) for i in range(300)}
    N, R = sum(rates.values()), 10
    num, den = 5 * N, 4 * R
    assert max(rates.values()) < fractions.Fraction(num, den)
    pl = O.build_plan(_keys_from_rates(rates), R, 8, num, den)
    assert (pl.adm_k == 1).all()
    pl2 = O.build_plan(_keys_from_rates(rates), R, 8, num, den, variant="NOREPL")
    assert pl.members.tolist() == pl2.members.tolist()


def _graham_instance(rng, m, n):
    jobs = rng.integers(1, 60, size=n).tolist()
    return jobs


@pytest.mark.parametrize("trial", range(40))
def test_lpt_within_graham_bound_of_brute_force(trial):
    # With every k_b = 1 and a uniform start, the placement is Graham's LPT list
    # schedule (sec. 3.1 cites Graham 1969); its makespan is within
    # (4/3 - 1/(3m)) of the optimum, found here by exhaustive search.
    rng = np.random.default_rng(1000 + trial)
    m = int(rng.integers(2, 5))
    n = int(rng.integers(1, 10))
    jobs = _graham_instance(rng, m, n)
    rates = {100 + i: j for i, j in enumerate(jobs)}
    N = sum(jobs)
    pl = O.build_plan(_keys_from_rates(rates), m, n, 10 ** 9, 1, init_load=np.zeros(m, np.uint64))
    assert pl.n_adm == n and (pl.adm_k == 1).all()
    makespan = int(pl.load.max())
    best = None
    for assign in itertools.product(range(m), repeat=n):
        L = [0] * m
        for j, a in zip(jobs, assign):
            L[a] += j
        best = max(L) if best is None else min(best, max(L))
    assert fractions.Fraction(makespan) <= (fractions.Fraction(4, 3) - fractions.Fraction(1, 3 * m)) * best
    assert int(pl.load.sum()) == N


def test_random_placement_is_uniform_and_deterministic():
    rates = {i: 1000 - i for i in range(64)}
    keys = _keys_from_rates(rates)
    R = 8
    counts = np.zeros(R)
    first = np.zeros(R)
    for seed in range(60):
        pl = O.build_plan(keys, R, 8, 10, 1, variant="RANDOM", seed=seed)
        again = O.build_plan(keys, R, 8, 10, 1, variant="RANDOM", seed=seed)
        assert pl.members.tolist() == again.members.tolist()
        for a in range(pl.n_adm):
            mem = pl.members[pl.koff[a]:pl.koff[a + 1]]
            assert len(set(mem.tolist())) == len(mem)
        counts += np.bincount(pl.members, minlength=R)
        first += np.bincount(pl.members[pl.koff[:-1]], minlength=R)
    # every key takes all R destinations here, so the ORDER must be uniform too:
    # which destination comes first (and so gets the larger job) is uniform.
    assert (counts == counts[0]).all()
    exp = first.sum() / R
    chi2 = float(((first - exp) ** 2 / exp).sum())
    assert chi2 < 30.0   # 7 dof; p ~ 1e-4
    other = O.build_plan(keys, R, 8, 10, 1, variant="RANDOM", seed=1, epoch=1)
    assert other.members.tolist() != O.build_plan(keys, R, 8, 10, 1, variant="RANDOM", seed=1).members.tolist()


def test_init_load_override_and_empty():
    pl = O.build_plan(np.zeros(0, np.uint64), 4, 2, 1, 1)
    assert pl.n_adm == 0 and pl.U == 0 and pl.load.tolist() == [0, 0, 0, 0]
    keys = _keys_from_rates({5: 3, 6: 2})
    pl = O.build_plan(keys, 3, 1, 100, 1, init_load=np.array([9, 0, 4], np.uint64))
    assert pl.members.tolist() == [1, 1] and pl.load.tolist() == [9, 5, 4]
    with pytest.raises(ValueError):
        O.build_plan(keys, 0, 1, 1, 1)
