"""Pins for the oracle's token-weighted (byte-aware) LRU replay (CPU only).

The byte-aware variant of the shadow-replay gate (sec. 3.1 and 6 mention byte
budgets; the replay model is this library's reading): each destination's cache
holds whole prefixes, most recent first, while their prefix tokens sum to at
most the capacity and there are at most 1024 of them.  The oracle simulates
every capacity on its own, by the textbook rule.  The pins: a hand-worked
trace; equal prefix sizes reduce it to the prefix-count LRU (itself pinned by
Mattson stack distances); and, when every key has one prefix length (as in
every trace here), a brute-force characterisation written without any cache
state -- a request hits iff its key was seen before and the prefix tokens of
the distinct keys used since its previous access, plus its own, fit the
capacity (and there are at most 1024 of them) -- which also shows that one
simulation at the largest capacity decides every smaller one.  A hand trace
pins the textbook rule when a key's length changes, where that shortcut fails.
"""
import numpy as np
import pytest

import oracle as O


def _run(keys, plen, caps, tokens=True, R=1, dest=None):
    n = len(keys)
    rp = O.Replay(1, R, caps, tokens=tokens)
    d = np.zeros((1, n), np.uint16) if dest is None else np.asarray(dest, np.uint16).reshape(1, n)
    ctr = rp.step(np.asarray(keys, np.uint64), np.asarray(plen, np.uint32), np.full(n, 64, np.uint32), d)
    return ctr.copy(), rp


def test_hand_trace():
    # capacity 5000 tokens: 1(2000) miss [1]; 2(3000) miss [2 1] = 5000; 1 hit [1 2];
    # 3(60) miss [3 1 2] = 5060 -> evict 2 -> [3 1]; 1 hit [1 3]; 2(3000) miss [2 1 3] = 5060
    # -> evict 3 -> [2 1].  Capacity 100: every prefix but key 3's is larger than the cache;
    # 3 enters, then 1 pushes both out.  Capacity 2000: [1]; 2 alone overflows and leaves
    # [] ; 1 miss [1]; 3 -> [3 1] = 2060 -> [3]; 1 miss [1 3] -> [1]; 2 -> [] .
    ctr, rp = _run([1, 2, 1, 3, 1, 2], [2000, 3000, 2000, 60, 2000, 3000], [5000, 100, 2000])
    hits = ctr[0, :, 0, 1].tolist()
    assert hits == [2, 0, 0]
    assert ctr[0, 0, 0].tolist() == [6, 2, 4000, 6 * 64 + 12060, 6 * 64 + 12060 - 4000]
    assert rp.state(0, 0, 0).tolist() == [2, 1]
    assert rp.state(0, 1, 0).tolist() == [] and rp.state(0, 2, 0).tolist() == []


@pytest.mark.parametrize("size,k", [(100, 1), (100, 3), (7, 12), (1, 40)])
def test_equal_sizes_reduce_to_prefix_count_lru(size, k):
    rng = np.random.default_rng(size + k)
    keys = rng.integers(0, 3 * k + 5, 3000)
    plen = np.full(keys.size, size)
    for extra in (0, size - 1):  # any capacity in [k * size, (k + 1) * size) holds exactly k prefixes
        ct, rt = _run(keys, plen, [k * size + extra])
        ce, re_ = _run(keys, plen, [k], tokens=False)
        assert (ct[..., [0, 1, 2, 4]] == ce[..., [0, 1, 2, 4]]).all()
        assert rt.state(0, 0, 0).tolist() == re_.state(0, 0, 0).tolist()


def _brute_hits(keys, plen, cap, max_entries=1024):
    """Hit iff seen before and the distinct keys used since (with their latest sizes) plus the
    key's own previous size fit the capacity, with at most max_entries prefixes."""
    hits = []
    for i, x in enumerate(keys):
        prev = None
        for j in range(i - 1, -1, -1):
            if keys[j] == x:
                prev = j
                break
        if prev is None:
            hits.append(False)
            continue
        latest = {}
        for j in range(prev + 1, i):
            latest[keys[j]] = plen[j]  # later accesses overwrite: latest size
        total = sum(latest.values()) + plen[prev]
        hits.append(total <= cap and len(latest) + 1 <= max_entries)
    return hits


@pytest.mark.parametrize("seed", range(5))
def test_brute_force_characterisation_all_capacities(seed):
    rng = np.random.default_rng(seed)
    nk = int(rng.integers(3, 40))
    keys = rng.integers(0, nk, 400).tolist()
    size_of = rng.integers(1, 3000 if seed % 2 else 300, nk)  # one prefix length per key
    plen = [int(size_of[k]) for k in keys]
    caps = [1, 500, 2999, 6000, 20000, 10 ** 6]
    ctr, _ = _run(keys, plen, caps)
    for c, cap in enumerate(caps):
        want = _brute_hits(keys, plen, cap)
        assert int(ctr[0, c, 0, 1]) == sum(want)
        assert int(ctr[0, c, 0, 2]) == sum(p for p, h in zip(plen, want) if h)
    hits = ctr[0, :, 0, 1]
    assert all(hits[i] <= hits[i + 1] for i in range(len(caps) - 1))  # inclusion


def test_changed_length_follows_the_textbook_rule():
    # Outside the one-length-per-key domain the oracle still applies the textbook rule to
    # each capacity: 1(4) then 2(8) at capacity 10 evicts 1; 2 coming back with length 2
    # leaves [2] (tokens 2), and 1 is a miss -- an evicted prefix does not come back
    # because another one shrank (so the longest-fitting-prefix rule needs fixed lengths).
    ctr, rp = _run([1, 2, 2, 1], [4, 8, 2, 4], [10])
    assert ctr[0, 0, 0, 1] == 1 and rp.state(0, 0, 0).tolist() == [1, 2]


def test_entry_limit_of_1024_prefixes():
    # 1500 distinct one-token prefixes, then the first ones again: a huge token capacity
    # still keeps only the 1024 most recent prefixes
    keys = list(range(1500)) + list(range(1500))
    plen = [1] * len(keys)
    ctr, rp = _run(keys, plen, [10 ** 9])
    want = _brute_hits(keys, plen, 10 ** 9)
    assert int(ctr[0, 0, 0, 1]) == sum(want) == 0  # each key comes back after 1499 others
    assert len(rp.state(0, 0, 0)) == 1024
    keys = list(range(1000)) + list(range(1000))
    ctr, rp = _run(keys, [1] * 2000, [10 ** 9])
    assert int(ctr[0, 0, 0, 1]) == 1000


def test_destinations_are_independent():
    rng = np.random.default_rng(9)
    keys = rng.integers(0, 30, 600)
    plen = rng.integers(100, 900, 600)
    dest = rng.integers(0, 3, 600)
    ctr, _ = _run(keys, plen, [2500], R=3, dest=dest)
    for r in range(3):
        m = dest == r
        ce, _ = _run(keys[m], plen[m], [2500])
        assert (ctr[0, 0, r] == ce[0, 0, 0]).all()
