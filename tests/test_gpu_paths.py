"""GPU: the TMA-staged kernels and the register kernel give identical results.

Streams with 16-byte aligned bases and rows of at least 512 bytes go through
the shared-memory (cp.async.bulk) kernel when they move bytes, and through
the plain-load tile kernel (k_hash) when they are only fingerprinted; a
context created with PCS_DISABLE_TMA=1 sends everything through the register
kernel.  All must agree with each other and with the oracle, byte for byte.
"""
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_bytes, np_view, u64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ctx_reg():
    old = os.environ.get("PCS_DISABLE_TMA")
    os.environ["PCS_DISABLE_TMA"] = "1"
    try:
        c = pcs.Context(0)
    finally:
        if old is None:
            del os.environ["PCS_DISABLE_TMA"]
        else:
            os.environ["PCS_DISABLE_TMA"] = old
    yield c
    c.close()


def test_fingerprints_agree(ctx, ctx_reg, dev):
    g = torch.Generator().manual_seed(12)
    sizes = [0, 16, 4096, 16384, 16384 + 16, 5 * 16384 + 4096, 1 << 20, (3 << 20) + 48, 100,
             16384 * 3 + 7]
    bufs = [torch.randint(0, 256, (n,), generator=g, dtype=torch.uint8).to(dev) for n in sizes]
    a = u64(ctx.fingerprint(bufs))
    b = u64(ctx_reg.fingerprint(bufs))
    assert a == b == [oracle.fingerprint(np_bytes(x)) for x in bufs]


def _kv_records(c, kv, dev, starts):
    kp, vp, pt, meta = kv.k_pool.to(dev), kv.v_pool.to(dev), kv.page_table.to(dev), kv.meta.to(dev)
    sess = [pcs.kv_session(s, meta[s], kp, vp, pt[s], starts[s], kv.window)
            for s in range(kv.sessions)]
    snaps = c.checkpoint(sess)
    recs = [c.record(x).numpy().copy() for x in snaps]
    # Restore into a fresh pool and read back the logical rows.
    pt2 = synth.page_permutation(5, kv.sessions, kv.layers, kv.window // kv.page_rows).to(dev)
    k2, v2, m2 = torch.zeros_like(kp), torch.zeros_like(vp), torch.zeros_like(meta)
    c.restore(snaps, [pcs.kv_session(s, m2[s], k2, v2, pt2[s], pcs.PCS_RING_START_FROM_SNAPSHOT,
                                     kv.window) for s in range(kv.sessions)], verify=True)
    for x in snaps:
        c.delete(x)
    torch.cuda.synchronize()
    j = torch.arange(kv.window)
    outs = []
    for s in range(kv.sessions):
        slot = (starts[s] + j) % kv.window
        pg = pt2[s].long().cpu()[:, slot // kv.page_rows]
        outs.append((k2.cpu()[pg, slot % kv.page_rows], v2.cpu()[pg, slot % kv.page_rows]))
    return recs, outs


def test_kv_paths_agree(ctx, ctx_reg, dev):
    kv = synth.kv(seed=61, sessions=3, layers=4, heads=16, head_dim=64, window=1024, page_rows=16)
    starts = [0, 9, 1000]
    ra, oa = _kv_records(ctx, kv, dev, starts)
    rb, ob = _kv_records(ctx_reg, kv, dev, starts)
    for s in range(kv.sessions):
        ref = oracle.pack(oracle.kv_session(s, kv.meta[s].numpy(), np_view(kv.k_pool),
                                            np_view(kv.v_pool), kv.page_table[s].numpy(),
                                            starts[s], kv.window, kv.page_rows, kv.row_bytes))
        assert np.array_equal(ra[s], ref) and np.array_equal(rb[s], ref), s
        j = torch.arange(kv.window)
        slot = (starts[s] + j) % kv.window
        pg = kv.page_table[s].long()[:, slot // kv.page_rows]
        want_k = kv.k_pool[pg, slot % kv.page_rows]
        assert torch.equal(oa[s][0], want_k) and torch.equal(ob[s][0], want_k)


def test_bank_rows_paths_agree(ctx, ctx_reg, dev):
    # 1 KiB keys and 32 KiB latent rows (TMA path) and 48-byte rows (register).
    b = synth.banks(62, 6, 1, 200, 512, torch.bfloat16, (16, 32, 32), torch.bfloat16)
    small = torch.randint(0, 256, (sum(b.n), 48), dtype=torch.uint8)
    for s in range(b.sessions):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        kept = torch.arange(0, hi - lo, 3, dtype=torch.int32)
        keys, vals = b.keys[lo:hi].to(dev), b.values[lo:hi].to(dev)
        sm = small[lo:hi].to(dev)
        kd = kept.to(dev)
        sess = pcs.Session(s, pcs.PCS_KIND_BANK, [
            pcs.contig_section(pcs.PCS_SEC_KEPT_IDX, kd, dim0=kd.numel()),
            pcs.rows_section(pcs.PCS_SEC_KEYS, keys, kd),
            pcs.rows_section(pcs.PCS_SEC_VALUES, vals.reshape(vals.shape[0], -1), kd),
            pcs.rows_section(9, sm, kd)], keep=[keys, vals, sm, kd])
        recs = []
        for c in (ctx, ctx_reg):
            snap = c.checkpoint([sess])[0]
            recs.append(c.record(snap).numpy().copy())
            c.delete(snap)
        sp = oracle.SessionSpec(s, oracle.KIND_BANK)
        kn = kept.numpy()
        sp.contig(oracle.SEC_KEPT_IDX, oracle.DT_I32, kn, dim0=kn.size)
        kh = np_view(b.keys[lo:hi])
        sp.rows(oracle.SEC_KEYS, oracle.DT_BF16, kh, kh.shape[1] * 2, kn, dim0=kn.size,
                dim1=kh.shape[1] * 2)
        vh = np.ascontiguousarray(np_view(b.values[lo:hi]).reshape(hi - lo, -1))
        sp.rows(oracle.SEC_VALUES, oracle.DT_BF16, vh, vh.shape[1] * 2, kn, dim0=kn.size,
                dim1=vh.shape[1] * 2)
        smh = small[lo:hi].numpy()
        sp.rows(9, oracle.DT_U8, smh, 48, kn, dim0=kn.size, dim1=48)
        ref = oracle.pack(sp)
        assert np.array_equal(recs[0], ref) and np.array_equal(recs[1], ref), s


def test_timing_reports_both_kernels(ctx, dev):
    ctx.timing(True)
    x = [torch.zeros(1 << 20, dtype=torch.uint8, device=dev),
         torch.zeros((1 << 20) + 1, dtype=torch.uint8, device=dev)[1:]]
    ctx.fingerprint(x)
    t = ctx.kernel_times()
    ctx.timing(False)
    assert t["k_hash"][0] == 1 and t["k_stream<hash>"][0] == 1
    assert t["k_finalize<hash>"][0] == 1


def test_small_unaligned_sources_in_large_calls(ctx, ctx_reg, dev):
    # A call past the small-call size mixes both kernels: the aligned
    # buffer goes through the TMA kernel, sections off a 16-byte boundary
    # (sources and restore targets) through the register kernel, in one call.
    g = torch.Generator().manual_seed(31)
    big = torch.randint(0, 256, (3 << 20,), generator=g, dtype=torch.uint8).to(dev)
    pool = torch.randint(0, 256, (1 << 18,), generator=g, dtype=torch.uint8).to(dev)
    views, off = [big], 0
    for n in [1, 3, 4, 15, 16, 17, 100, 511, 4095, 4096, 4097, 8191, 8192, 8193]:
        for shift in (1, 2, 4, 8, 12):
            off += shift
            views.append(pool[off:off + n])
            off += n
    assert off <= pool.numel()
    want = [oracle.fingerprint(np_bytes(x)) for x in views]
    assert u64(ctx.fingerprint(views)) == want
    assert u64(ctx_reg.fingerprint(views)) == want
    # Checkpoint: one big aligned section and small unaligned ones per session.
    sess = []
    for s in range(6):
        secs = [pcs.contig_section(pcs.PCS_SEC_OBS, big[s << 18:(s + 1) << 18])]
        secs += [pcs.contig_section(pcs.PCS_SEC_KEPT_IDX, v) for v in views[1 + s::6]]
        sess.append(pcs.Session(s, pcs.PCS_KIND_MARKOV, secs, keep=[big, pool]))
    snaps = ctx.checkpoint(sess)
    for s, sn in enumerate(snaps):
        sp = oracle.SessionSpec(s, oracle.KIND_MARKOV)
        sp.contig(pcs.PCS_SEC_OBS, oracle.DT_U8, np_bytes(big[s << 18:(s + 1) << 18]))
        for v in views[1 + s::6]:
            sp.contig(pcs.PCS_SEC_KEPT_IDX, oracle.DT_U8, np_bytes(v))
        assert np.array_equal(ctx.record(sn).numpy(), oracle.pack(sp)), s
    # Restore into targets that are themselves off a 16-byte boundary.
    tpool = torch.zeros(1 << 18, dtype=torch.uint8, device=dev)
    tb = torch.zeros(6 << 18, dtype=torch.uint8, device=dev)
    tg, toff, tv = [], 3, []
    for s in range(6):
        secs = [pcs.contig_section(pcs.PCS_SEC_OBS, tb[s << 18:(s + 1) << 18])]
        for v in views[1 + s::6]:
            t = tpool[toff:toff + v.numel()]
            toff += v.numel() + 5
            tv.append((t, v))
            secs.append(pcs.contig_section(pcs.PCS_SEC_KEPT_IDX, t))
        tg.append(pcs.Session(s, pcs.PCS_KIND_MARKOV, secs, keep=[tb, tpool]))
    ctx.restore(snaps, tg, verify=True)
    torch.cuda.synchronize()
    assert torch.equal(tb, big[:6 << 18])
    for t, v in tv:
        assert torch.equal(t, v)
    for sn in snaps:
        ctx.delete(sn)


@pytest.mark.parametrize("sessions", [64, 2000, 3400])
def test_markov_batches_static_and_shared_tma_kernels(ctx, dev, sessions):
    """One checkpoint call of many Markov sessions, below and above the size
    at which the TMA kernel stops handing out its last tiles at run time
    (launches of fewer than 64 tiles per warp share them; on 152 SMs 2,000
    sessions are 50,000 tiles, 3,400 sessions 85,000): every record equals
    the oracle's, byte for byte, and a verified restore brings every byte back."""
    g = torch.Generator(device=dev).manual_seed(77 + sessions)
    obs = torch.randint(0, 256, (sessions, 3, 256, 256), generator=g, device=dev,
                        dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (sessions, 2), generator=g, device=dev, dtype=torch.int64)
    arr = ctx.session_array([pcs.markov_session(s, obs[s], rng[s]) for s in range(sessions)])
    hs = ctx.checkpoint_raw(arr, sessions)
    obs_h, rng_h = obs.cpu().numpy(), rng.cpu().numpy().view(np.uint64)
    for s in range(sessions):
        ref = oracle.pack(oracle.markov_session(s, obs_h[s], rng_h[s]))
        assert np.array_equal(ctx.record(pcs.Snapshot(ctx, hs[s])).numpy(), ref), s
    o2, r2 = torch.zeros_like(obs), torch.zeros_like(rng)
    tarr = ctx.session_array([pcs.markov_session(s, o2[s], r2[s]) for s in range(sessions)])
    ctx.restore_raw(hs, sessions, tarr, verify=1)
    torch.cuda.synchronize()
    assert torch.equal(o2, obs) and torch.equal(r2, rng)
    ctx.delete_raw(hs, sessions)
