"""Pins of the oracle's content fingerprint and classification (CPU only).

The paper prints no hash (Sec. 4 only requires that must-snapshot be decided
by whether a recompute reproduces a buffer).  PCSFP64-v1 is a frozen reading,
so these tests pin the oracle to what that definition must satisfy: the
published SplitMix64 vectors for its mixer, the per-word bijection that makes
any single-bit change visible, order and length sensitivity, the lane
partition of a chunk, and the aligned-group decomposition of the tree, plus
brute force by an independent top-down restatement of the tree.
"""
import os
import random

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
M64 = 2**64 - 1


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def test_fmix_is_splitmix64():
    # Published SplitMix64 outputs for state 0 (Steele, Lea & Flood 2014).
    expected = [int(r[0], 16) for r in _read_golden("splitmix64_seed0.txt")]
    x, got = 0, []
    for _ in expected:
        x = (x + 0x9E3779B97F4A7C15) & M64
        got.append(oracle.fmix(x))
    assert got == expected


def _tree_top_down(items):
    """Independent restatement: root = comb(T(first 2^k), T(rest)), 2^k < n <= 2^(k+1)."""
    n = len(items)
    if n == 1:
        return items[0]
    h = 1
    while 2 * h < n:
        h *= 2
    return oracle.comb(_tree_top_down(items[:h]), _tree_top_down(items[h:]))


@pytest.mark.parametrize("n", list(range(1, 40)) + [63, 64, 65, 100, 257])
def test_tree_matches_top_down_restatement(n):
    rnd = random.Random(n)
    items = [rnd.getrandbits(64) for _ in range(n)]
    assert oracle.tree(items) == _tree_top_down(items)


@pytest.mark.parametrize("n", [1, 2, 3, 31, 32, 33, 64, 100, 1000, 4097])
@pytest.mark.parametrize("group", [2, 4, 32, 64])
def test_tree_aligned_group_decomposition(n, group):
    # Reducing aligned groups of 2^m items first (a GPU block's share), then
    # the list of group roots, gives the same root: scheduling-independent.
    rnd = random.Random(n * 131 + group)
    items = [rnd.getrandbits(64) for _ in range(n)]
    roots = [oracle.tree(items[g:g + group]) for g in range(0, n, group)]
    assert oracle.tree(roots) == oracle.tree(items)


def test_tree_is_order_sensitive():
    items = [1, 2, 3, 4, 5]
    assert oracle.tree(items) != oracle.tree([2, 1, 3, 4, 5])
    assert oracle.tree(items) != oracle.tree([1, 2, 3, 5, 4])


def test_lane_tree_equals_list_tree():
    data = np.arange(4096, dtype=np.uint32).view(np.uint8)[:4096]
    lanes = [oracle.lane_value(data, 0, l) for l in range(32)]
    assert oracle.chunk_hash(data, 0) == oracle.tree(lanes)


def test_lane_partition_of_a_chunk():
    # Lane l owns 16-byte segments l, l+32, ..., l+224: changing segment s
    # changes lane s mod 32's value and no other lane's.
    rnd = np.random.default_rng(5)
    data = rnd.integers(0, 256, 4096, dtype=np.uint8)
    base = [oracle.lane_value(data, 0, l) for l in range(32)]
    for seg in [0, 1, 31, 32, 33, 100, 224, 255]:
        d2 = data.copy()
        d2[16 * seg + 3] ^= 0x40
        now = [oracle.lane_value(d2, 0, l) for l in range(32)]
        changed = [l for l in range(32) if now[l] != base[l]]
        assert changed == [seg % 32], (seg, changed)


@pytest.mark.parametrize("L", [1, 7, 16, 37, 4096, 4097])
def test_every_single_bit_flip_changes_fp(L):
    # Every step is a bijection of each u64 word given the others, so any
    # single-bit change must change the fingerprint -- with certainty.
    rnd = np.random.default_rng(L)
    data = rnd.integers(0, 256, L, dtype=np.uint8)
    fp0 = oracle.fingerprint(data)
    bits = range(8 * L) if L <= 64 else sorted(
        set(rnd.integers(0, 8 * L, 300).tolist()) | set(range(8 * L - 64, 8 * L)))
    for b in bits:
        d2 = data.copy()
        d2[b // 8] ^= np.uint8(1 << (b % 8))
        assert oracle.fingerprint(d2) != fp0, b


def test_any_single_word_change_changes_fp():
    rnd = np.random.default_rng(11)
    data = rnd.integers(0, 2**63, 3 * 512 + 7, dtype=np.uint64)
    fp0 = oracle.fingerprint(data)
    for _ in range(200):
        i = int(rnd.integers(0, data.size))
        d2 = data.copy()
        d2[i] = np.uint64((int(d2[i]) + int(rnd.integers(1, 2**62))) & M64)
        assert oracle.fingerprint(d2) != fp0


def test_length_enters_the_fingerprint():
    # Bytes past L read as zero, so a trailing zero byte changes nothing but
    # L; the fingerprint must still differ (length finalisation).
    for L in [0, 1, 15, 4095, 4096, 8191]:
        a = np.full(L, 9, dtype=np.uint8)
        b = np.concatenate([a, np.zeros(1, dtype=np.uint8)])
        assert oracle.fingerprint(a) != oracle.fingerprint(b), L
        assert oracle.chunk_hash(a, 0) == oracle.chunk_hash(b, 0)


def test_tail_reads_as_zero_padding():
    rnd = np.random.default_rng(3)
    L = 2 * 4096 + 100
    data = rnd.integers(0, 256, L, dtype=np.uint8)
    padded = np.zeros(3 * 4096, dtype=np.uint8)
    padded[:L] = data
    for c in range(3):
        assert oracle.chunk_hash(data, c) == oracle.chunk_hash(padded, c, L=3 * 4096)
    C = oracle.n_chunks(L)
    assert C == 3
    xs = [oracle.chunk_hash(padded, c, L=3 * 4096) for c in range(3)]
    assert oracle.fingerprint(data) == oracle.fmix(oracle.tree(xs) ^ ((L * 0x9E3779B97F4A7C15) & M64))


def test_chunk_position_enters_the_hash():
    # Identical chunk contents at different positions hash differently, so
    # swapping two equal chunks with a third cannot go unnoticed.
    block = np.full(4096, 0xAB, dtype=np.uint8)
    data = np.concatenate([block, block])
    assert oracle.chunk_hash(data, 0) != oracle.chunk_hash(data, 1)
    rnd = np.random.default_rng(4)
    a = rnd.integers(0, 256, 4096, dtype=np.uint8)
    b = rnd.integers(0, 256, 4096, dtype=np.uint8)
    assert oracle.fingerprint(np.concatenate([a, b])) != oracle.fingerprint(np.concatenate([b, a]))


def test_n_chunks():
    assert [oracle.n_chunks(L) for L in [0, 1, 4095, 4096, 4097, 8192]] == [1, 1, 1, 1, 2, 2]


def test_known_answers_frozen():
    # Regression anchor written by tests/golden/make_fp_kat.py (oracle only).
    for L, fp in _read_golden("fp_kat.txt"):
        L = int(L)
        data = ((131 * np.arange(L, dtype=np.uint64) + 7) % 256).astype(np.uint8)
        assert oracle.fingerprint(data) == int(fp, 16), L


def test_fingerprint_many_matches_single():
    rnd = np.random.default_rng(8)
    bufs = [rnd.integers(0, 256, n, dtype=np.uint8) for n in [0, 1, 100, 5000, 9000]]
    many = oracle.fingerprint_many(bufs)
    assert [int(x) for x in many] == [oracle.fingerprint(b) for b in bufs]


def test_classify_matches_seeded_ground_truth():
    # Sec. 4 step 1 at epsilon = 0: must-snapshot iff the recompute did not
    # reproduce the buffer.  Ground truth: which buffers got a bit flipped.
    import torch
    from paper_2607_21686_gb300 import synth
    sw = synth.sweep(seed=123, n=40, lo=64, hi=1 << 16)
    def raw(t):
        return t.contiguous().view(torch.uint8).numpy()
    before = oracle.fingerprint_many([raw(t) for t in sw.before])
    after = oracle.fingerprint_many([raw(t) for t in sw.after])
    flags = oracle.classify(before, after)
    assert flags.tolist() == [1 if f else 0 for f in sw.flipped]
    assert sum(sw.flipped) == 12
