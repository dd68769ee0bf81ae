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


def test_many_handles_in_random_order(ctx, dev):
    """Thousands of live handles made by several calls and forks, deleted in
    a random order between further calls: the live count, each surviving
    handle's info and record, and the refusal of handles that were never
    made all hold while handle objects are reused."""
    import ctypes
    rnd = np.random.default_rng(5)
    base = ctx.stats().live_snapshots
    t = torch.arange(64, dtype=torch.uint8, device=dev)
    arr = ctx.session_array([_sess(t, sid=s) for s in range(3000)])
    live = {}
    for rounds in range(4):
        hs = ctx.checkpoint_raw(arr, 3000)
        kids = ctx.fork_raw(hs, 3000)
        for i in range(3000):
            live[hs[i]] = i
            live[kids[i]] = i
        ctx.sync()
        assert ctx.stats().live_snapshots == base + len(live)
        doomed = rnd.choice(sorted(live), size=len(live) // 2, replace=False)
        batch = (ctypes.c_void_p * len(doomed))(*[int(h) for h in doomed])
        ctx.delete_raw(batch, len(doomed))
        for h in doomed:
            del live[int(h)]
        assert ctx.stats().live_snapshots == base + len(live)
    for h in rnd.choice(sorted(live), size=50, replace=False):
        snap = pcs.Snapshot(ctx, int(h))
        assert ctx.info(snap).session_id == live[int(h)]
        assert ctx.info(snap).n_sections == 1
        off = ctx.section(snap, 0).offset
        assert np.array_equal(ctx.record(snap).numpy()[off:off + 64], np.arange(64, dtype=np.uint8))
    for bad in (8, 1 << 40, max(live) + 8):
        with pytest.raises(pcs.PcsError) as e:
            ctx.info(pcs.Snapshot(ctx, bad))
        assert e.value.status == pcs.PCS_E_HANDLE
    rest = sorted(live)
    ctx.delete_raw((ctypes.c_void_p * len(rest))(*rest), len(rest))
    assert ctx.stats().live_snapshots == base
