"""Bounded device waits: a wait that can never end gives up and is reported.

Every wait inside the library's kernels (the TMA pipeline's mbarrier waits,
the grid barrier of the global threshold) is bounded by about two seconds of
SM clock; past the bound the kernel sets the timeout bit and returns, so a
stuck wait becomes PCS_E_TIMEOUT at the next pcs_sync instead of a hung GPU.
pcs_selftest_wait makes one thread wait, through those same helpers, for
something nothing provides (an mbarrier's second arrival, a flag nothing
writes).  No fault is injected: the wait simply runs out.
"""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs
from helpers import u64

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("which", [0, 1], ids=["mbarrier", "flag"])
def test_wait_that_never_ends_times_out_and_context_stays_usable(ctx, dev, which):
    t0 = time.perf_counter()
    ctx.selftest_wait(which)
    with pytest.raises(pcs.PcsError) as e:
        ctx.sync()
    took = time.perf_counter() - t0
    assert e.value.status == pcs.PCS_E_TIMEOUT
    assert 0.5 < took < 60.0, took  # the bound is about two seconds of SM clock
    # The error was cleared and the context works: a fingerprint against the oracle.
    g = torch.Generator().manual_seed(11 + which)
    x = torch.randint(0, 256, (3 * 4096 + 5,), generator=g, dtype=torch.uint8)
    fp = ctx.fingerprint([x.to(dev)])
    ctx.sync()
    assert u64(fp) == [oracle.fingerprint(x.numpy())]


def test_selftest_rejects_unknown_wait(ctx):
    with pytest.raises(pcs.PcsError) as e:
        ctx.selftest_wait(2)
    assert e.value.status == pcs.PCS_E_INVAL
    ctx.sync()  # nothing was enqueued
