"""The allocation-free key histogram, checked against the oracle's and the plan builder's.

cr_key_histogram_noalloc serves callers that cannot allocate device memory
when they call in (device memory owned by another runtime's pool, or a
latency-critical path that cannot afford cudaMalloc).  It must give exactly
the oracle's histogram (and the one cr_build_plans computes) for the same
keys, on repeated calls (its scratch array is shared and keeps the previous
call's contents), and reject inputs larger than its fixed scratch.  This file
is collected last so that a failure here never hides the results of the
other tests.
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytestmark = [pytest.mark.gpu, pytest.mark.skip(reason="needs a CUDA GPU")]
else:
    pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0)


@pytest.fixture(scope="module")
def P():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_19677_gb300 as P
    L = P.lib()
    f = L.cr_key_histogram_noalloc
    f.argtypes = [ctypes.c_void_p, ctypes.c_uint64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                  ctypes.c_void_p]
    f.restype = ctypes.c_int
    return P


def _keys(seed, nkeys, n):
    rng = np.random.default_rng(seed)
    pool = rng.integers(0, 2**64, size=nkeys, dtype=np.uint64)
    pool[:3] = [0, 2**64 - 1, 2**64 - 2]          # extreme values, incl. the table's empty marker
    w = rng.pareto(1.1, size=nkeys) + 1e-3
    idx = rng.choice(nkeys, size=n, p=w / w.sum())
    return pool[idx]


def _noalloc(P, keys):
    n = keys.size
    dk = torch.from_numpy(keys.view(np.int64)).to(DEV)
    uk = torch.full((max(n, 1),), -7, dtype=torch.int64, device=DEV)
    uc = torch.full((max(n, 1),), -7, dtype=torch.int64, device=DEV)
    U = torch.full((1,), -7, dtype=torch.int64, device=DEV)
    stream = torch.cuda.current_stream(DEV).cuda_stream
    st = P.lib().cr_key_histogram_noalloc(dk.data_ptr(), n, uk.data_ptr(),
                                          uc.data_ptr(), U.data_ptr(), stream)
    assert st == P.CR_OK, P.lib().cr_last_error(None)
    torch.cuda.synchronize()
    u = int(U.item())
    return uk[:u].cpu().numpy().view(np.uint64), uc[:u].cpu().numpy().view(np.uint64)


def _reference(P, ctx, keys):
    dk = torch.from_numpy(keys.view(np.int64)).to(DEV)
    pl = P.build_plan(ctx, dk, P.plan_params(8, 4, max(keys.size, 1), 32))
    got = pl.export()
    return got["ukey"], got["ucnt"]


def test_noalloc_histogram_matches_plan_builder_twice(P):
    import oracle as O
    ctx = P.Context(0)
    for seed, nkeys, n in ((1, 3000, 60000), (2, 50, 700)):   # second call smaller: stale contents must not leak
        keys = _keys(seed, nkeys, n)
        uk, uc = _noalloc(P, keys)
        ok, oc = O.histogram(keys)                # the oracle's (key ascending, count)
        assert uk.size == ok.size and (uk == ok).all() and (uc == oc).all()
        rk, rc = _reference(P, ctx, keys)
        assert uk.size == rk.size and (uk == rk).all() and (uc == rc).all()
        assert int(uc.sum()) == n
    ctx.close()


def test_noalloc_histogram_limits(P):
    L = P.lib()
    d = torch.zeros(1, dtype=torch.int64, device=DEV)
    stream = torch.cuda.current_stream(DEV).cuda_stream
    st = L.cr_key_histogram_noalloc(d.data_ptr(), P.CR_NOALLOC_MAX_KEYS + 1, d.data_ptr(), d.data_ptr(),
                                    d.data_ptr(), stream)
    assert st == P.CR_EINVAL and b"CR_NOALLOC_MAX_KEYS" in L.cr_last_error(None)
    # empty input: U = 0
    U = torch.full((1,), 5, dtype=torch.int64, device=DEV)
    assert L.cr_key_histogram_noalloc(None, 0, None, None, U.data_ptr(), stream) == P.CR_OK
    torch.cuda.synchronize()
    assert int(U.item()) == 0
