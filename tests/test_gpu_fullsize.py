"""Parity at full interval sizes, in the launch configuration bench.py times.

For each of the five synthetic configurations the first two control intervals
run through the device pipeline exactly as the benchmark runs them (planner
on its own stream, batches of 1024).  The oracle then checks, at full size:
  - every request's routing key (the oracle hashes each distinct key's
    prefix once; requests that carry the same key share their prefix);
  - the complete plans interval 1 was routed with (built from interval 0);
  - the complete destinations, in both intervals, of every plan-based replica
    (CacheRoute and its ablations: the method's own dispatch through the
    device table) and of one power-of-two-choices replica;
  - the complete replay counters of those replicas after both intervals;
and every replica's counters satisfy request conservation, LRU inclusion
across capacities and prefill = prompt - hit tokens.  The oracle runs one
replica per thread (each call is plain single-threaded C).
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


def oracle_keys(trace, key_ids):
    """Routing key of every request, the oracle hashing each distinct key's prefix once."""
    ids = np.unique(np.concatenate(key_ids))
    kv = np.empty(ids.size, np.uint64)
    chunk = 50000
    for a in range(0, ids.size, chunk):
        tok, off, pl = tg.prefix_spans(trace, ids[a:a + chunk])
        kv[a:a + chunk] = O.hash_prefixes(tok, off, pl)
    return [kv[np.searchsorted(ids, k)] for k in key_ids]


@pytest.mark.parametrize("name", ["tiny", "70b", "8b", "burst", "large"])
def test_fullsize_two_intervals(P, name):
    from paper_2608_19677_gb300.pipeline import Pipeline
    cfg = tg.CONFIGS[name]
    tr = tg.Trace(cfg)
    nint = min(2, cfg.n_intervals)
    ivs = [tr.interval(t) for t in range(nint)]
    ctx = P.Context(0)
    pipe = Pipeline(ctx, cfg.R, cfg.W, cfg.caps, cfg.replicas, tr.qcap, batch_B=1024,
                    max_n=max(iv.n for iv in ivs), overlap=True)
    dkeys, dests, plans_used = [], [], []
    for t, iv in enumerate(ivs):
        tok, off = tg.arena_device(tr, iv, 4, device=DEV)
        plen = torch.from_numpy(iv.plen.view(np.int32)).to(DEV)
        slen = torch.from_numpy(iv.slen.view(np.int32)).to(DEV)
        keys = pipe.interval(t, tok, off, plen, slen, iv.g0, plan_next=t + 1 < nint)
        dkeys.append(keys.cpu().numpy().view(np.uint64).copy())
        pipe.wait_last()
        dests.append(pipe.last_dest.cpu().numpy().view(np.uint16).copy())
        plans_used.append([pl.export() for pl in pipe.last_plans])
        del tok, off
    pipe.finish()
    pipe.sync()
    ctr = pipe.ctr.cpu().numpy().view(np.uint64).copy()

    # ---- keys: every request, via the oracle's hash of its key's prefix ----------
    okeys = oracle_keys(tr, [iv.key_id for iv in ivs])
    for t in range(nint):
        assert (dkeys[t] == okeys[t]).all(), f"interval {t}: keys differ"

    # ---- the plan interval 1 was routed with (interval 0 for a single interval) ---
    tp = nint - 1
    plan_from = okeys[tp - 1] if tp > 0 else okeys[0]
    per_rep, built = OP.plans_for_interval(tr, plan_from, tp)
    for (v, s), got in zip(pipe.plan_keys, plans_used[tp]):
        ref = built[(v, s)]
        assert got["n_adm"] == ref.n_adm and got["sum_k"] == ref.sum_k and got["cold"] == ref.cold
        assert (got["adm_key"] == ref.adm_key).all()
        assert (got["members"] == ref.members).all() and (got["jobs"] == ref.jobs).all()
        assert (got["load"] == ref.load).all()

    # ---- complete destinations and replay of every plan-based replica and one P2C replica ----
    reps = cfg.replicas
    plan_based = [i for i, (p, _) in enumerate(reps) if OP.VARIANT_OF.get(p) is not None]
    p2c = [i for i, (p, _) in enumerate(reps) if p == "P2C"][:1]
    checked = plan_based + p2c
    assert plan_based, "every configuration has CacheRoute replicas"
    plans_t = [OP.plans_for_interval(tr, okeys[t - 1] if t > 0 else okeys[0], t)[0] for t in range(nint)]

    def one_replica(i):
        pol, seed = reps[i]
        pol = OP.ROUTE_AS.get(pol, pol)
        orp = O.Replay(1, cfg.R, cfg.caps)
        bad = []
        for t in range(nint):
            d, _ = O.route([plans_t[t][i]], [pol], [seed], cfg.R, okeys[t], ivs[t].g0, 1024)
            if not (dests[t][i] == d[0]).all():
                bad.append(f"interval {t}: {int((dests[t][i] != d[0]).sum())} destinations differ")
            orp.step(okeys[t], ivs[t].plen, ivs[t].slen, d)
        if not (ctr[i] == orp.ctr[0]).all():
            bad.append("replay counters differ")
        return i, bad

    import concurrent.futures as cf
    import os
    with cf.ThreadPoolExecutor(max_workers=min(len(checked), os.cpu_count() or 1)) as ex:
        for i, bad in ex.map(one_replica, checked):
            assert not bad, f"replica {reps[i]}: {'; '.join(bad)}"

    # ---- properties of every replica -------------------------------------------
    n_all = sum(iv.n for iv in ivs)
    prompt_all = sum(int(iv.plen.astype(np.int64).sum() + iv.slen.astype(np.int64).sum()) for iv in ivs)
    for r in range(len(reps)):
        for c in range(len(cfg.caps)):
            assert int(ctr[r, c, :, 0].sum()) == n_all
            assert int(ctr[r, c, :, 3].sum()) == prompt_all
        assert (ctr[r, :, :, 4] == ctr[r, :, :, 3] - ctr[r, :, :, 2]).all()
        order = np.argsort(cfg.caps)
        for a, b in zip(order[:-1], order[1:]):
            assert (ctr[r, a, :, 1] <= ctr[r, b, :, 1]).all()
    ctx.close()
