"""Pins for the oracle's bounded-load comparison policy (CPU only).

The policy is consistent hashing with bounded loads (Mirrokni, Thorup and
Zadimoghaddam, SODA 2018) at epsilon = 0.25 (sec. 4).  The ring layout is this
library's reading: destination d owns V points, point (d, v) being SplitMix64
output number d*V + v from the ring seed.  The pins are the published
SplitMix64 stream, a brute-force walk that orders every point by its clockwise
distance from the key (no sorted ring, no binary search, no wrap-around code),
keys placed exactly on a point and past the last point through the inverse of
the mixing function, the bound max load <= ceil((1 + eps) m / R) after every
request, and the reduction to plain consistent hashing when no destination is
at its bound.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as O

M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15
C1, C2 = 0xBF58476D1CE4E5B9, 0x94D049BB133111EB


def _published(golden_dir):
    vals = []
    with open(os.path.join(golden_dir, "splitmix64_seed0.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                vals.append(int(line, 16))
    return vals


def _unxorshift(y, s):
    x = y
    for _ in range(64 // s + 1):
        x = y ^ (x >> s)
    return x & M64


def _fmix64_inverse(z):
    z = _unxorshift(z, 31)
    z = (z * pow(C2, -1, 1 << 64)) & M64
    z = _unxorshift(z, 27)
    z = (z * pow(C1, -1, 1 << 64)) & M64
    return _unxorshift(z, 30)


def _points(R, V, seed):
    return [(O.fmix64((seed + (k + 1) * GAMMA) & M64), k // V) for k in range(R * V)]


def _brute_chwbl(R, V, ring_seed, key_seed, keys, B, load0):
    """Walk every point in order of clockwise distance from the key's position."""
    pts = _points(R, V, ring_seed)
    L = [int(x) for x in load0]
    dest = []
    for b0 in range(0, len(keys), B):
        snap = list(L)
        m = sum(snap)
        cap = math.ceil(Fraction(5 * (m + 1), 4 * R))  # ceil((1 + 1/4) (m + 1) / R)
        for key in keys[b0:b0 + B]:
            h = O.fmix64(int(key) ^ key_seed)
            order = sorted(pts, key=lambda po: ((po[0] - h) & M64, po[1]))
            d = next(o for _, o in order if snap[o] < cap)
            dest.append(d)
            L[d] += 1
    return dest, L


def test_inverse_mix_is_exact():
    rng = np.random.default_rng(5)
    for z in [0, 1, M64, GAMMA] + [int(x) for x in rng.integers(0, 1 << 63, 50, dtype=np.int64)]:
        assert O.fmix64(_fmix64_inverse(z)) == z


def test_ring_seed0_is_the_published_splitmix64_stream(golden_dir):
    pub = _published(golden_dir)
    pt, ow = O.Ring(3, 1, 0).export()
    assert pt.tolist() == sorted(pub)
    assert ow.tolist() == [pub.index(p) for p in sorted(pub)]
    pt1, ow1 = O.Ring(1, 3, 0).export()
    assert pt1.tolist() == sorted(pub) and ow1.tolist() == [0, 0, 0]


@pytest.mark.parametrize("R,V,seed", [(5, 7, 123), (2, 64, 2 ** 63 + 5), (40, 3, 1)])
def test_ring_is_the_sorted_point_set(R, V, seed):
    pt, ow = O.Ring(R, V, seed).export()
    want = sorted(_points(R, V, seed))
    assert pt.tolist() == [p for p, _ in want]
    assert ow.tolist() == [o for _, o in want]
    assert np.bincount(ow, minlength=R).tolist() == [V] * R


def _edge_keys(R, V, ring_seed, key_seed, rng, n):
    """Random keys plus keys exactly on ring points, just past a point, and past the last point."""
    pts = sorted(p for p, _ in _points(R, V, ring_seed))
    ks = [int(x) for x in rng.integers(0, 1 << 63, n, dtype=np.int64)]
    for p in pts[:3] + pts[-2:]:
        ks.append(_fmix64_inverse(p) ^ key_seed)
        ks.append(_fmix64_inverse((p + 1) & M64) ^ key_seed)
    if pts[-1] < M64:
        ks.append(_fmix64_inverse(M64) ^ key_seed)  # wraps to the first point
    ks.append(_fmix64_inverse(0) ^ key_seed)
    rng.shuffle(ks)
    return np.array(ks, dtype=np.uint64)


@pytest.mark.parametrize("R,V,B,start", [(1, 4, 1, "zero"), (3, 2, 1, "zero"), (7, 5, 1, "random"),
                                         (7, 5, 3, "random"), (16, 4, 32, "zero"), (5, 3, 1000, "random"),
                                         (12, 1, 1, "skewed")])
def test_chwbl_matches_clockwise_brute_force(R, V, B, start):
    rng = np.random.default_rng(R * 100 + V * 10 + B)
    ring_seed, key_seed = 77 + R, 991
    hot = rng.integers(0, 1 << 63, 6, dtype=np.int64)
    keys = _edge_keys(R, V, ring_seed, key_seed, rng, 120)
    keys = np.concatenate([keys, hot[rng.integers(0, 6, 150)].astype(np.uint64)])
    if start == "zero":
        load0 = np.zeros(R, np.uint64)
    elif start == "random":
        load0 = rng.integers(0, 40, R).astype(np.uint64)
    else:
        load0 = np.zeros(R, np.uint64)
        load0[: R // 2] = 500
    ring = O.Ring(R, V, ring_seed)
    dest, load = O.route([None], ["CHWBL"], [key_seed], R, keys, g0=0, B=B, load=load0[None, :],
                         rings=[ring])
    want, wl = _brute_chwbl(R, V, ring_seed, key_seed, keys, B, load0)
    assert dest[0].tolist() == want
    assert load[0].tolist() == wl


@pytest.mark.parametrize("R,V", [(2, 8), (9, 16), (64, 4)])
def test_chwbl_sequential_load_bound(R, V):
    # With batch_B = 1 no destination ever exceeds ceil((1 + 1/4) m / R) after m requests.
    rng = np.random.default_rng(R)
    keys = rng.integers(0, 40, 3000).astype(np.uint64) * np.uint64(0x9E3779B97F4A7C15)  # few hot keys
    dest, load = O.route([None], ["CHWBL"], [3], R, keys, g0=0, B=1, rings=[O.Ring(R, V, 4)])
    L = np.zeros(R, np.int64)
    for m, d in enumerate(dest[0].tolist(), start=1):
        L[d] += 1
        assert L.max() <= math.ceil(Fraction(5 * m, 4 * R))
    assert load[0].tolist() == L.tolist()


def test_chwbl_unsaturated_is_consistent_hashing():
    # One batch from zero loads: cap = ceil(5 / (4R)) = 1 > 0 for R >= 2, so every
    # request goes to the owner of the nearest point clockwise of its position.
    R, V, rs, ks = 11, 9, 5, 6
    rng = np.random.default_rng(0)
    keys = _edge_keys(R, V, rs, ks, rng, 300)
    dest, _ = O.route([None], ["CHWBL"], [ks], R, keys, g0=0, B=len(keys), rings=[O.Ring(R, V, rs)])
    pts = _points(R, V, rs)
    for key, d in zip(keys.tolist(), dest[0].tolist()):
        h = O.fmix64(key ^ ks)
        assert d == min(pts, key=lambda po: ((po[0] - h) & M64, po[1]))[1]


def test_chwbl_skips_destinations_at_the_bound():
    R, V, rs, ks = 4, 1, 8, 2
    pts = sorted(_points(R, V, rs))
    key = _fmix64_inverse(pts[0][0]) ^ ks  # lands exactly on the first point
    load0 = np.zeros(R, np.uint64)
    load0[pts[0][1]] = 10  # m = 10: cap = ceil(55 / 16) = 4
    dest, _ = O.route([None], ["CHWBL"], [ks], R, np.array([key], np.uint64), g0=0, B=1,
                      load=load0[None, :], rings=[O.Ring(R, V, rs)])
    assert dest[0, 0] == pts[1][1]
    load0[pts[1][1]] = 4  # m = 14: cap = ceil(75 / 16) = 5 > 4
    dest, _ = O.route([None], ["CHWBL"], [ks], R, np.array([key], np.uint64), g0=0, B=1,
                      load=load0[None, :], rings=[O.Ring(R, V, rs)])
    assert dest[0, 0] == pts[1][1]
    load0[pts[1][1]] = 5  # m = 15: cap = 5 -> skipped too
    dest, _ = O.route([None], ["CHWBL"], [ks], R, np.array([key], np.uint64), g0=0, B=1,
                      load=load0[None, :], rings=[O.Ring(R, V, rs)])
    assert dest[0, 0] == pts[2][1]


def test_chwbl_needs_a_matching_ring():
    with pytest.raises(ValueError):
        O.route([None], ["CHWBL"], [1], 4, np.arange(5, dtype=np.uint64), g0=0, B=1)
    with pytest.raises(ValueError):
        O.route([None], ["CHWBL"], [1], 4, np.arange(5, dtype=np.uint64), g0=0, B=1, rings=[O.Ring(5, 2, 0)])
