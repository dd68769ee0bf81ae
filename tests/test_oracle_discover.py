"""Pins of the oracle's discovery procedure, distance and read classification.

Sec. 4 (procedure FINGERPRINT): necessity by leave-one-out, sufficiency of the
necessary set, greedy redundancy fallback for correlated or mutually
recomputable buffers.  Sec. 3 ("A distinction the implementation forced"): a
buffer is PCS iff restore reads it.  The pins use synthetic probes whose PCS
is known by construction, a byte-level bitmap restatement of the overlap test,
and the paper's own sizes for the state / witness split.
"""
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# -- distance ---------------------------------------------------------------

def test_mismatch_closed_forms():
    rnd = np.random.default_rng(0)
    a = rnd.integers(0, 256, 1000, dtype=np.uint8)
    assert oracle.mismatch(a, a.copy()) == 0
    assert oracle.mismatch(a, a ^ 0xFF) == 1000
    b = a.copy()
    b[[3, 500, 999]] ^= 1
    assert oracle.mismatch(a, b) == 3
    assert oracle.mismatch(a, a[:990]) == 10
    assert oracle.mismatch(a[:0], a[:7]) == 7
    # Any dtype: bytes are compared.
    x = np.arange(10, dtype=np.float32)
    y = x.copy()
    y[4] = -y[4]
    assert oracle.mismatch(x, y) == 1  # only the sign byte differs


# -- state versus witness ---------------------------------------------------

def _bitmap_flags(bufs, reads, space):
    touched = np.zeros(space, dtype=bool)
    for r, n in reads:
        touched[r:r + n] = True
    return np.array([1 if n and touched[b:b + n].any() else 0 for b, n in bufs], dtype=np.uint8)


@pytest.mark.parametrize("seed", range(30))
def test_read_classification_matches_byte_bitmap(seed):
    rnd = np.random.default_rng(seed)
    space = 600
    bufs = [(int(rnd.integers(0, 550)), int(rnd.integers(0, 50))) for _ in range(12)]
    reads = [(int(rnd.integers(0, 590)), int(rnd.integers(0, 10))) for _ in range(int(rnd.integers(0, 15)))]
    assert oracle.classify_reads(bufs, reads).tolist() == _bitmap_flags(bufs, reads, space).tolist()


def test_read_classification_edges():
    bufs = [(100, 10), (110, 10), (105, 0), (200, 50), (210, 5)]
    assert oracle.classify_reads(bufs, [(110, 1)]).tolist() == [0, 1, 0, 0, 0]
    assert oracle.classify_reads(bufs, [(109, 1)]).tolist() == [1, 0, 0, 0, 0]
    assert oracle.classify_reads(bufs, [(109, 2)]).tolist() == [1, 1, 0, 0, 0]
    assert oracle.classify_reads(bufs, [(90, 10), (120, 80)]).tolist() == [0, 0, 0, 0, 0]
    assert oracle.classify_reads(bufs, [(105, 0), (212, 1)]).tolist() == [0, 0, 0, 1, 1]
    assert oracle.classify_reads(bufs, []).tolist() == [0] * 5


def _golden():
    rows, totals, witness = [], {}, {}
    with open(os.path.join(GOLDEN, "state_witness.txt")) as f:
        for line in f:
            p = line.split()
            if not p or p[0].startswith("#"):
                continue
            if p[0] == "total":
                totals[p[1]] = int(p[2])
            elif p[0] == "with_witness":
                witness[p[1]] = float(p[2])
            else:
                rows.append((p[0], p[1], int(p[2]), int(p[3])))
    return rows, totals, witness


def test_state_witness_split_reproduces_table_sizes():
    rows, totals, witness = _golden()
    for model in totals:
        mine = [r for r in rows if r[0] == model]
        addr, bufs, reads = 4096, [], []
        for _, _, nbytes, is_read in mine:
            bufs.append((addr, nbytes))
            if is_read:  # restore reads every byte of it, in 4 KiB pieces
                reads += [(a, min(4096, addr + nbytes - a)) for a in range(addr, addr + nbytes, 4096)]
            addr += nbytes + 256
        flags = oracle.classify_reads(bufs, reads)
        assert flags.tolist() == [r[3] for r in mine]
        assert sum(n for (_, n), f in zip(bufs, flags) if f) == totals[model]
        if model in witness:
            assert round(sum(n for _, n in bufs) / 1e6, 2) == witness[model]


# -- discovery ----------------------------------------------------------------

def _weighted_probe(weights, need):
    # D = sum of the weights of needed components that were not snapshotted.
    return lambda keep: sum(w for w, n, k in zip(weights, need, keep) if n and not k)


def test_independent_components_are_found_in_k_plus_one_probes():
    need = [1, 0, 1, 0, 0, 1]
    pcs, probes, ok = oracle.discover(6, _weighted_probe([5, 5, 1, 9, 9, 2], need), 0)
    assert pcs.tolist() == need and probes == 7 and ok


def test_tolerance_drops_cheap_components():
    need = [1, 1, 1]
    pcs, _, ok = oracle.discover(3, _weighted_probe([10, 3, 7], need), 3)
    assert pcs.tolist() == [1, 0, 1] and ok


def test_mutually_recomputable_pair_takes_the_fallback():
    # Components 1 and 3 recompute each other: D > 0 only if both are missing.
    def probe(keep):
        d = 4 * (not keep[0]) + 6 * (not keep[4])
        return d + (8 if not keep[1] and not keep[3] else 0)
    pcs, probes, ok = oracle.discover(5, probe, 0)
    # Necessity finds {0, 4}; sufficiency fails; one fallback round tries
    # 1, 2, 3 and keeps the first of the two that fix it.
    assert pcs.tolist() == [1, 1, 0, 0, 1] and ok
    assert probes == 5 + 1 + 3


def test_fallback_prefers_the_larger_reduction():
    # 1 and 2 partly stand in for each other: missing both costs 10, missing
    # only 1 costs 1, missing only 2 costs 2.  Both pass the fallback's bar
    # (eps = 2), but adding 2 reduces D more, so it is the one added.
    def probe(keep):
        d = 0 if keep[0] else 5
        if not keep[1] and not keep[2]:
            d += 10
        elif not keep[1]:
            d += 1
        elif not keep[2]:
            d += 2
        return d
    pcs, probes, ok = oracle.discover(3, probe, 2)
    assert pcs.tolist() == [1, 0, 1] and ok and probes == 3 + 1 + 2


def test_no_consistent_set_reports_it():
    pcs, probes, ok = oracle.discover(3, lambda keep: 1, 0)
    assert pcs.tolist() == [1, 1, 1] and not ok
    pcs, probes, ok = oracle.discover(0, lambda keep: 0, 0)
    assert pcs.size == 0 and probes == 1 and ok
