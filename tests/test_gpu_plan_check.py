"""GPU: with PCS_CHECK=1 every plan is checked on the host before launch
(node slots inside the node array, work lists covering each stream's tasks
once, addressable layouts, payloads inside their records).  Every kind of
call plans within those invariants and gives the same results as a context
without the checks."""
import ctypes
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_bytes, np_view, u64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx_chk():
    old = os.environ.get("PCS_CHECK")
    os.environ["PCS_CHECK"] = "1"
    try:
        c = pcs.Context(0)
    finally:
        if old is None:
            del os.environ["PCS_CHECK"]
        else:
            os.environ["PCS_CHECK"] = old
    yield c
    c.close()


def test_checked_fingerprints(ctx_chk, dev):
    g = torch.Generator().manual_seed(21)
    # tiny (one fused launch), unaligned, TMA-sized and a 5 MiB buffer whose
    # 640 tile nodes take a reduction level
    sizes = [0, 17, 4096, (1 << 20) + 48, 5 << 20]
    bufs = [torch.randint(0, 256, (n + 1,), generator=g, dtype=torch.uint8).to(dev) for n in sizes]
    views = [b[1:] if i == 1 else b[:-1] for i, b in enumerate(bufs)]
    assert u64(ctx_chk.fingerprint(views)) == [oracle.fingerprint(np_bytes(v)) for v in views]
    assert u64(ctx_chk.fingerprint(views[:2])) == [oracle.fingerprint(np_bytes(v)) for v in views[:2]]


def test_checked_checkpoint_restore_fork(ctx_chk, dev):
    n = 16
    g = torch.Generator(device=dev).manual_seed(22)
    obs = torch.randint(0, 256, (n, 3, 256, 256), generator=g, device=dev, dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (n, 2), generator=g, device=dev, dtype=torch.int64)
    big = torch.randint(0, 256, (5 << 20,), generator=g, device=dev, dtype=torch.uint8)
    sess = [pcs.markov_session(s, obs[s], rng[s]) for s in range(n)]
    for place in (pcs.PCS_PLACE_DEVICE, pcs.PCS_PLACE_PINNED_HOST):
        snaps = ctx_chk.checkpoint(sess, placement=place)
        for s in (0, n - 1):
            ref = oracle.pack(oracle.markov_session(s, obs[s].cpu().numpy(),
                                                    rng[s].cpu().numpy().view(np.uint64)))
            assert np.array_equal(ctx_chk.record(snaps[s]).numpy(), ref)
        kids = [ctx_chk.fork(x) for x in snaps[:3]]
        o2, r2 = torch.zeros_like(obs), torch.zeros_like(rng)
        ctx_chk.restore(snaps, [pcs.markov_session(s, o2[s], r2[s]) for s in range(n)], verify=True)
        torch.cuda.synchronize()
        assert torch.equal(o2, obs) and torch.equal(r2, rng)
        for x in snaps + kids:
            ctx_chk.delete(x)
    # One section of 640 tiles: a reduction level before finalisation.
    one = pcs.Session(7, pcs.PCS_KIND_MARKOV,
                      [pcs.contig_section(pcs.PCS_SEC_OBS, big, dim0=big.numel())], keep=[big])
    snap = ctx_chk.checkpoint([one])[0]
    assert ctx_chk.section(snap, 0).fp == oracle.fingerprint(big.cpu().numpy())
    ctx_chk.delete(snap)


def test_checked_banks_and_kv(ctx_chk, dev):
    b = synth.banks_config2(seed=23, sessions=8)
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]].to(dev) for s in range(b.sessions)]
    vals = [b.values[b.entry_off[s]:b.entry_off[s + 1]].to(dev) for s in range(b.sessions)]
    banks = ctx_chk.banks_array(keys, [b.queries[s].to(dev) for s in range(b.sessions)],
                                512 + b.value_bytes)
    params = ctx_chk.params(pcs.PCS_K_FIXED, k_max=128)
    ks = ctx_chk.prune_counts(banks, b.sessions, params)
    koff = np.concatenate([[0], np.cumsum(ks)]).astype(int)
    kept = torch.empty(int(koff[-1]), dtype=torch.int32, device=dev)
    ctx_chk.prune(banks, b.sessions, params, kept)
    sess = [pcs.bank_session(s, keys[s], vals[s], kept[koff[s]:koff[s + 1]])
            for s in range(b.sessions)]
    snaps = ctx_chk.checkpoint(sess)
    kept_h = kept.cpu().numpy()
    for s in range(b.sessions):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        ref = oracle.pack(oracle.bank_session(s, np_view(b.keys[lo:hi]), np_view(b.values[lo:hi]),
                                              np.ascontiguousarray(kept_h[koff[s]:koff[s + 1]]),
                                              oracle.DT_F16, oracle.DT_BF16))
        assert np.array_equal(ctx_chk.record(snaps[s]).numpy(), ref), s
    for x in snaps:
        ctx_chk.delete(x)
    kv = synth.kv(seed=24, sessions=3, layers=4, heads=4, head_dim=64, window=1024, page_rows=16)
    kp, vp, pt, meta = kv.k_pool.to(dev), kv.v_pool.to(dev), kv.page_table.to(dev), kv.meta.to(dev)
    snaps = ctx_chk.checkpoint([pcs.kv_session(s, meta[s], kp, vp, pt[s], kv.ring_start[s],
                                               kv.window) for s in range(kv.sessions)])
    for s in range(kv.sessions):
        ref = oracle.pack(oracle.kv_session(s, kv.meta[s].numpy(), np_view(kv.k_pool),
                                            np_view(kv.v_pool), kv.page_table[s].numpy(),
                                            kv.ring_start[s], kv.window, kv.page_rows,
                                            kv.row_bytes))
        assert np.array_equal(ctx_chk.record(snaps[s]).numpy(), ref), s
    hs = (ctypes.c_void_p * kv.sessions)(*[x.handle for x in snaps])
    plan = ctx_chk.plan_restore(hs, kv.sessions,
                                ctx_chk.session_array([pcs.kv_session(s, meta[s], kp, vp, pt[s],
                                                                      pcs.PCS_RING_START_FROM_SNAPSHOT,
                                                                      kv.window)
                                                       for s in range(kv.sessions)]), verify=2)
    ctx_chk.plan_run(plan)
    ctx_chk.sync()
    ctx_chk.plan_destroy(plan)
    for x in snaps:
        ctx_chk.delete(x)
