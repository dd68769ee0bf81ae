"""GPU: snapshot memory is reused only after the work that reads it.

A restore is queued, its snapshot deleted at once, and a checkpoint of other
bytes issued on a second stream takes the freed memory: the restore must
still see the original record (the freed range carries the restore's event,
and the new allocation waits for it on its own stream).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs
from helpers import np_bytes

pytestmark = pytest.mark.gpu


def _sess(t, sid=1):
    return pcs.Session(sid, pcs.PCS_KIND_MARKOV,
                       [pcs.contig_section(pcs.PCS_SEC_OBS, t, dim0=t.numel())], keep=[t])


def test_delete_while_restore_pending_then_reuse_on_other_stream(ctx, dev):
    n = 256 << 20
    g = torch.Generator(device=dev).manual_seed(77)
    x = torch.randint(0, 256, (n,), generator=g, device=dev, dtype=torch.uint8)
    z = torch.randint(0, 256, (n,), generator=g, device=dev, dtype=torch.uint8)
    y = torch.zeros_like(x)
    s1 = torch.cuda.current_stream()
    s2 = torch.cuda.Stream()
    for _ in range(3):
        a = ctx.checkpoint([_sess(x)])[0]
        torch.cuda.synchronize()
        ctx.restore([a], [_sess(y)], verify=2, stream=s1)
        ctx.delete(a)                                  # restore still queued
        with torch.cuda.stream(s2):
            b = ctx.checkpoint([_sess(z, 2)], stream=s2)[0]  # may take a's memory
        torch.cuda.synchronize()
        ctx.sync()
        assert torch.equal(y, x)
        assert ctx.section(b, 0).fp == oracle.fingerprint(np_bytes(z))
        ctx.delete(b)
        y.zero_()
