"""Host-side logic on the CPU: configuration transforms of the bench, the trace generator's
token capacities, and agreement between the device pipeline and the oracle pipeline on how
policies map to plan variants and route policies."""
import numpy as np

import bench
import oracle.pipeline as OP
import paper_2608_19677_gb300 as P
import paper_2608_19677_gb300.pipeline as PP
import tracegen as tg


def test_policy_maps_agree():
    assert PP.VARIANT_OF == OP.VARIANT_OF
    assert PP.ROUTE_AS == OP.ROUTE_AS
    for pol, var in PP.VARIANT_OF.items():
        assert var in P.VARIANT
        assert PP.ROUTE_AS.get(pol, pol) in P.POLICY
    # every policy the generator names has a library id, and the ids agree with the oracle's
    for name, pid in tg.POLICY_IDS.items():
        assert P.POLICY[name] == pid
    import oracle as O
    assert O.POLICY == P.POLICY
    assert set(O.VARIANT) == set(P.VARIANT) and all(O.VARIANT[k] == P.VARIANT[k] for k in O.VARIANT)


def test_token_capacities():
    assert tg.CONFIGS["70b"].token_lru().caps == [24576]
    large = tg.CONFIGS["large"].token_lru()
    assert large.caps == [c * 2048 for c in tg.CONFIGS["large"].caps] and large.lru_tokens
    eightb = tg.CONFIGS["8b"].token_lru()
    assert eightb.caps == [64 * (1024 + 4096) // 2]
    assert tg.CONFIGS["70b"].token_lru().token_lru().caps == [24576]  # idempotent


def test_bench_config_transforms():
    base = tg.CONFIGS["70b"]
    cfg = bench.with_policies(base, bench.parse_args([]))
    assert cfg is base
    cfg = bench.with_policies(base, bench.parse_args(["--policies", "CR,CHWBL", "--token-lru", "--trace-seed", "7"]))
    assert cfg.policies == ["CR", "CHWBL"] and cfg.seeds == base.seeds
    assert cfg.lru_tokens and cfg.caps == [24576] and cfg.trace_seed == 7
    assert [p for p, _ in cfg.replicas] == ["CR"] * 5 + ["CHWBL"] * 5
    w = bench.workload_config(cfg, 1, fresh=True)
    assert w["batch_B"] == 1 and w["lru_capacity_unit"] == "prefix tokens" and "own keys" in w["plans_from"]


def test_rings_follow_replicas():
    import dataclasses
    cfg = dataclasses.replace(tg.CONFIGS["tiny"], policies=["CR", "CHWBL", "P2C"], seeds=[3, 4])
    rings = OP.rings_for(cfg)
    assert [r is not None for r in rings] == [p == "CHWBL" for p, _ in cfg.replicas]
    assert [r.seed for r in rings if r is not None] == [3, 4]
    pt, ow = rings[2].export()
    assert np.all(np.diff(pt.astype(np.float64)) >= 0) and np.bincount(ow, minlength=cfg.R).tolist() == [cfg.vnodes] * cfg.R
