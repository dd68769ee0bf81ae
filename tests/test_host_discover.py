"""The library's discovery procedure (host code, no GPU) against the oracle's.

pcs_discover runs the Sec. 4 procedure over a caller probe; here the probes
are plain Python functions with known answers, so the library and the oracle
must agree on the PCS flags, the number of probes and consistency.
"""
import numpy as np
import pytest

import oracle
from paper_2607_21686_gb300 import pcs


def _random_probe(seed):
    # Components in groups: a group costs its weight when none of its members
    # is kept (a group of two or more is a set of mutually recomputable
    # buffers); some components belong to no group (derivable).
    rnd = np.random.default_rng(seed)
    k = int(rnd.integers(0, 9))
    groups, free = [], list(rnd.permutation(k))
    while free and rnd.random() < 0.8:
        size = int(rnd.integers(1, 4))
        groups.append(([int(x) for x in free[:size]], int(rnd.integers(1, 20))))
        free = free[size:]
    noise = int(rnd.integers(0, 3))

    def probe(keep):
        d = sum(w for g, w in groups if not any(keep[i] for i in g))
        # A cross term so that the greedy choice depends on the reduction.
        return d + noise * sum(1 for i in range(k) if not keep[i])
    return k, probe, int(rnd.integers(0, 6))


@pytest.mark.parametrize("seed", range(60))
def test_library_discovery_matches_oracle(seed):
    k, probe, eps = _random_probe(seed)
    got = pcs.discover(k, probe, eps)
    want = oracle.discover(k, probe, eps)
    assert got[0] == want[0].tolist() and got[1] == want[1] and got[2] == want[2]


def test_probe_failure_stops_the_procedure():
    calls = []

    def probe(keep):
        calls.append(list(keep))
        if len(calls) == 3:
            raise ValueError("model crashed")
        return 0
    with pytest.raises(ValueError):
        pcs.discover(5, probe, 0)
    assert len(calls) == 3
