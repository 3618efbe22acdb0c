"""Pins for the oracle's mixing functions and prefix-span key (CPU only).

The key definition is this library's reading (the paper routes on an opaque,
possibly salted business key, sec. 3.1 and the supplement's data-handling
note); these tests tie the oracle's arithmetic to published values (SplitMix64
outputs, numpy's Philox4x64-10) and to structural identities a wrong index,
sign or dropped term would break.
"""
import os

import numpy as np
import pytest

import oracle as O
import tracegen as tg

M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15


def _splitmix_published(golden_dir):
    vals = []
    with open(os.path.join(golden_dir, "splitmix64_seed0.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                vals.append(int(line, 16))
    return vals


def test_fmix64_matches_published_splitmix64(golden_dir):
    pub = _splitmix_published(golden_dir)
    assert len(pub) == 3
    for i, v in enumerate(pub):
        assert O.fmix64((i + 1) * GAMMA) == v


@pytest.mark.parametrize("key", [(0, 0), (5, 7), (M64, 1), (0x0123456789ABCDEF, 0xFEDCBA9876543210)])
@pytest.mark.parametrize("ctr0", [0, 10, 1 << 40])
def test_philox_matches_numpy(key, ctr0):
    # numpy's Philox bit generator emits philox(counter + 1, key) for state counter c.
    bg = np.random.Philox(key=np.array(key, dtype=np.uint64),
                         counter=np.array([ctr0, 3, 0, 9], dtype=np.uint64))
    ref = [int(x) for x in bg.random_raw(4)]
    assert O.philox4x64_10([ctr0 + 1, 3, 0, 9], list(key)) == ref


def test_philox_random123_zero_vector():
    # Known-answer vector for Philox4x64-10 with zero counter and key, as
    # produced by numpy's independent implementation one counter step earlier.
    bg = np.random.Philox(key=np.zeros(2, np.uint64), counter=np.full(4, M64, np.uint64))
    ref = [int(x) for x in bg.random_raw(4)]
    assert O.philox4x64_10([0, 0, 0, 0], [0, 0]) == ref


def test_hash_all_zero_span_is_header_plus_splitmix_stream(golden_dir):
    # With tokens all zero every word term is fmix64(salt + (i+1)*gamma): the
    # SplitMix64 output stream seeded with `salt`.  With salt 0 these are the
    # published outputs; the header term is fmix64(P) for P = 6, and
    # fmix64(P) is itself pinned below through P = gamma multiples.
    pub = _splitmix_published(golden_dir)
    h6 = O.hash_one(np.zeros(6, np.int32), salt=0)
    assert h6 == (O.fmix64(6) + sum(pub)) & M64
    h2 = O.hash_one(np.zeros(2, np.int32), salt=0)
    assert (h6 - h2) & M64 == (O.fmix64(6) - O.fmix64(2) + pub[1] + pub[2]) & M64
    # header via a salt that makes salt ^ P a gamma multiple: salt = gamma ^ P
    P = 2
    salt = GAMMA ^ P
    h = O.hash_one(np.zeros(P, np.int32), salt=salt)
    assert h == (pub[0] + O.fmix64((salt + GAMMA) & M64)) & M64


def test_hash_additive_by_position():
    # key = header + sum_i f_i(w_i): swapping word values between two prefixes
    # at two different positions satisfies H(u,x)+H(v,y) == H(u,y)+H(v,x).
    rng = np.random.default_rng(1)
    base = rng.integers(0, 128256, size=40).astype(np.int32)
    def with_words(i_val, j_val):
        t = base.copy()
        t[4:6] = i_val
        t[30:32] = j_val
        return O.hash_one(t, salt=77)
    u, v, x, y = ([1, 2], [3, 4], [5, 6], [7, 8])
    assert (with_words(u, x) + with_words(v, y)) & M64 == (with_words(u, y) + with_words(v, x)) & M64
    # ... but the same word at a different position contributes differently
    t1 = base.copy(); t1[4:6] = u; t1[30:32] = x
    t2 = base.copy(); t2[4:6] = x; t2[30:32] = u
    assert O.hash_one(t1, 77) != O.hash_one(t2, 77)


def test_hash_odd_length_and_padding():
    x = 123456
    h = O.hash_one(np.array([x], np.int32), salt=9)
    assert h == (O.fmix64(9 ^ 1) + O.fmix64(x ^ ((9 + GAMMA) & M64))) & M64
    # [x] and [x, 0] share the word but not the length
    assert O.hash_one(np.array([x, 0], np.int32), 9) != h


def test_hash_sensitivity():
    rng = np.random.default_rng(2)
    t = rng.integers(0, 128256, size=301).astype(np.int32)
    h = O.hash_one(t, 5)
    for j in [0, 1, 2, 150, 299, 300]:
        u = t.copy()
        u[j] ^= 1
        assert O.hash_one(u, 5) != h
    u = t.copy(); u[[10, 11]] = u[[11, 10]]
    assert O.hash_one(u, 5) != h
    assert O.hash_one(t, 6) != h
    assert O.hash_one(t[:300], 5) != h
    assert O.hash_one(np.zeros(0, np.int32), 3) == O.fmix64(3)


def test_hash_prefixes_reads_prefix_only():
    cfg = tg.CONFIGS["tiny"].scaled(300, 1)
    tr = tg.Trace(cfg)
    iv = tr.interval(0)
    for align in (1, 4):
        tok, off = tg.arena_host(tr, iv, align)
        keys = O.hash_prefixes(tok, off, iv.plen, salt=0)
        for i in [0, 1, 7, iv.n - 1]:
            pref = tg.prefix_tokens(tr, int(iv.key_id[i]))
            assert keys[i] == O.hash_one(pref, 0)
        # requests with the same business key get the same routing key
        for kid in np.unique(iv.key_id)[:20]:
            assert len(set(keys[iv.key_id == kid].tolist())) == 1
        # perturbing suffix tokens changes nothing
        tok2 = tok.copy()
        for i in range(iv.n):
            s = int(off[i]) + int(iv.plen[i])
            tok2[s:s + int(iv.slen[i])] += 1
        assert (O.hash_prefixes(tok2, off, iv.plen) == keys).all()


def test_no_collisions_on_tiny_trace():
    tr = tg.Trace(tg.CONFIGS["tiny"])
    iv = tr.interval(0)
    tok, off = tg.arena_host(tr, iv, 4)
    keys = O.hash_prefixes(tok, off, iv.plen)
    assert len(np.unique(keys)) == len(np.unique(iv.key_id))
