"""GPU parity: prune, checkpoint, fork, restore through the C ABI vs the oracle.

Records must equal the oracle's PCS1 records byte for byte; restored bytes
must equal the pre-checkpoint bytes after an excursion (I1); snapshots are
unaffected by later writes (I2); forks are independent (I3); records hold
exactly the selected sections (I4).  Scores agree with the oracle's fixed
order fp32 score bit for bit and with its fp64 cosine within 1e-3 relative;
kept sets are exact.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_bytes, np_view, u64

pytestmark = pytest.mark.gpu

SCORE_RTOL = 1e-3


# ---------------------------------------------------------------------------
# Markovian sessions (config 1 shape)
# ---------------------------------------------------------------------------

def test_markov_round_trip_and_record(ctx, dev):
    m = synth.markov(seed=synth.seed_for(1))
    obs_h, rng_h = m.obs.clone(), m.rng.clone()
    obs, rng = m.obs.to(dev), m.rng.to(dev)
    snap = ctx.checkpoint([pcs.markov_session(3, obs, rng)])[0]
    ref = oracle.pack(oracle.markov_session(3, obs_h.numpy(), rng_h.numpy().view(np.uint64)))
    assert np.array_equal(ctx.record(snap).numpy(), ref)
    info = ctx.info(snap)
    assert info.total_bytes == ref.size and info.n_sections == 2 and info.session_id == 3
    assert info.session_fp == oracle.record_header(ref)["session_fp"]
    # Section fps equal the stand-alone fingerprint of the live buffers.
    fps = u64(ctx.fingerprint([obs, rng]))
    assert [ctx.section(snap, i).fp for i in range(2)] == fps
    # Excursion overwrites both buffers; the snapshot is unaffected (I2).
    synth.excursion(m, seed=1234)
    obs.copy_(m.obs)
    rng.copy_(m.rng)
    assert np.array_equal(ctx.record(snap).numpy(), ref)
    ctx.restore([snap], [pcs.markov_session(3, obs, rng)], verify=True)
    torch.cuda.synchronize()
    assert torch.equal(obs.cpu(), obs_h) and torch.equal(rng.cpu(), rng_h)
    ctx.delete(snap)
    ctx.sync()


def test_rng_bit_flip_changes_session_fp(ctx, dev):
    m = synth.markov(seed=9)
    obs, rng = m.obs.to(dev), m.rng.to(dev)
    s0 = ctx.checkpoint([pcs.markov_session(0, obs, rng)])[0]
    rng.view(torch.uint8)[5] ^= 0x10
    s1 = ctx.checkpoint([pcs.markov_session(0, obs, rng)])[0]
    i0, i1 = ctx.info(s0), ctx.info(s1)
    assert i0.session_fp != i1.session_fp
    assert ctx.section(s0, 0).fp == ctx.section(s1, 0).fp
    assert ctx.section(s0, 1).fp != ctx.section(s1, 1).fp
    ctx.delete(s0)
    ctx.delete(s1)


def test_many_markov_sessions_one_call(ctx, dev):
    ms = [synth.markov(seed=100 + i, shape=(3, 17 + i, 31)) for i in range(40)]
    sess = [pcs.markov_session(i, m.obs.to(dev), m.rng.to(dev)) for i, m in enumerate(ms)]
    snaps = ctx.checkpoint(sess, placement=pcs.PCS_PLACE_PINNED_HOST)
    for i, (m, s) in enumerate(zip(ms, snaps)):
        ref = oracle.pack(oracle.markov_session(i, m.obs.numpy(), m.rng.numpy().view(np.uint64)))
        assert np.array_equal(ctx.record(s).numpy(), ref), i
    outs = [(torch.zeros_like(m.obs, device=dev), torch.zeros_like(m.rng, device=dev)) for m in ms]
    ctx.restore(snaps, [pcs.markov_session(i, o, r) for i, (o, r) in enumerate(outs)], verify=True)
    torch.cuda.synchronize()
    for m, (o, r) in zip(ms, outs):
        assert torch.equal(o.cpu(), m.obs) and torch.equal(r.cpu(), m.rng)
    for s in snaps:
        ctx.delete(s)


# ---------------------------------------------------------------------------
# Memory banks (config 2 shape, smaller / full)
# ---------------------------------------------------------------------------

def _bank_views(b, dev):
    keys, vals, qs = [], [], []
    for s in range(b.sessions):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        keys.append(b.keys[lo:hi].to(dev))
        vals.append(b.values[lo:hi].to(dev))
        qs.append(b.queries[s].to(dev))
    return keys, vals, qs


def _check_prune(ctx, b, keys, qs, params, dev):
    n = b.sessions
    banks = ctx.banks_array(keys, qs, keys[0].shape[1] * 2 + b.value_bytes)
    ks = ctx.prune_counts(banks, n, params)
    total = sum(b.n)
    kept = torch.empty(max(sum(ks), 1), dtype=torch.int32, device=dev)
    koff = torch.empty(n + 1, dtype=torch.int32, device=dev)
    scores = torch.empty(max(total, 1), dtype=torch.float32, device=dev)
    ctx.prune(banks, n, params, kept, koff, scores)
    ctx.sync()
    kept_h, koff_h, sc_h = kept.cpu().numpy(), koff.cpu().numpy(), scores.cpu().numpy()
    assert koff_h.tolist() == np.concatenate([[0], np.cumsum(ks)]).tolist()
    for s in range(n):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        s32, s64 = oracle.scores(np_view(b.queries[s]), np_view(b.keys[lo:hi]), want64=True)
        got = sc_h[lo:hi]
        assert np.array_equal(got.view(np.uint32), s32.view(np.uint32)), s
        np.testing.assert_allclose(got, s64, rtol=SCORE_RTOL, atol=1e-6)
        want = oracle.topk(s32, ks[s])
        assert kept_h[koff_h[s]:koff_h[s + 1]].tolist() == want.tolist(), s
    return ks, kept, koff


@pytest.mark.parametrize("rule", ["fixed", "fraction", "budget"])
def test_bank_prune_small(ctx, dev, rule):
    b = synth.banks(21, 12, 1, 300, 256, torch.float16, (16, 32, 32), torch.bfloat16)
    keys, vals, qs = _bank_views(b, dev)
    if rule == "fixed":
        p = ctx.params(pcs.PCS_K_FIXED, k_max=128)
    elif rule == "fraction":
        p = ctx.params(pcs.PCS_K_FRACTION, fraction=0.12)
    else:
        p = ctx.params(pcs.PCS_K_BUDGET, budget=sum(b.n) * (512 + b.value_bytes) // 3)
    _check_prune(ctx, b, keys, qs, p, dev)


def test_bank_prune_ties_and_degenerate(ctx, dev):
    # Duplicate keys (exact ties), a zero key (score 0), the query itself.
    D = 64
    g = torch.Generator().manual_seed(4)
    q = torch.randn(D, generator=g).half()
    base = torch.randn(5, D, generator=g).half()
    keys = torch.cat([base, base, torch.zeros(1, D).half(), q[None], -q[None], base[:2]])
    b = synth.Banks(n=[keys.shape[0]], entry_off=[0, keys.shape[0]], keys=keys,
                    values=torch.zeros(keys.shape[0], 16, dtype=torch.uint8), queries=q[None],
                    key_dim=D, value_bytes=16)
    for k in [0, 1, 3, 6, 7, 10, keys.shape[0], keys.shape[0] + 5]:
        p = ctx.params(pcs.PCS_K_FIXED, k_max=k)
        _check_prune(ctx, b, [keys.to(dev)], [q.to(dev)], p, dev)


@pytest.mark.parametrize("largest", [512, 513])
def test_prune_ties_at_every_bank_size(ctx, dev, largest):
    """Relevance pruning where every threshold falls in a run of exact ties:
    banks of 0, 1, 2, 31, 32, 33, 255, 511 and `largest` entries drawn from a
    few distinct keys, with zero keys (score 0) and negated queries (negative
    scores) among them; k from 0 to past n, and a fraction.  Scores, kept
    sets and offsets equal the oracle's."""
    D = 128
    g = torch.Generator().manual_seed(largest)
    sizes = [0, 1, 2, 31, 32, 33, 255, 511, largest, 0, 7]
    q = [torch.randn(D, generator=g).half() for _ in sizes]
    keys = []
    for i, n in enumerate(sizes):
        pool = torch.randn(5, D, generator=g).half()
        pool[1] = 0
        pool[2] = -q[i]
        pick = torch.randint(0, 5, (n,), generator=g)
        keys.append(pool[pick])
    n_tot = sum(sizes)
    b = synth.Banks(n=sizes, entry_off=np.concatenate([[0], np.cumsum(sizes)]).tolist(),
                    keys=torch.cat(keys), values=torch.zeros(n_tot, 16, dtype=torch.uint8),
                    queries=torch.stack(q), key_dim=D, value_bytes=16)
    kd = [x.to(dev) for x in keys]
    qd = [x.to(dev) for x in q]
    for k in [0, 1, 2, 17, 32, 100, 256, 511, 600]:
        _check_prune(ctx, b, kd, qd, ctx.params(pcs.PCS_K_FIXED, k_max=k), dev)
    _check_prune(ctx, b, kd, qd, ctx.params(pcs.PCS_K_FRACTION, fraction=0.37), dev)


def _bank_round_trip(ctx, b, dev, params, placement):
    keys, vals, qs = _bank_views(b, dev)
    ks, kept, koff = _check_prune(ctx, b, keys, qs, params, dev)
    koff_h = koff.cpu().tolist()
    sess = [pcs.bank_session(s, keys[s], vals[s], kept[koff_h[s]:koff_h[s + 1]])
            for s in range(b.sessions)]
    snaps = ctx.checkpoint(sess, placement=placement)
    kept_h = kept.cpu().numpy()
    kdt = oracle.DT_F16 if b.keys.dtype == torch.float16 else oracle.DT_BF16
    vdt = oracle.DT_BF16 if b.values.dtype == torch.bfloat16 else oracle.DT_U8
    refs = []
    for s in range(b.sessions):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        kp = np.ascontiguousarray(kept_h[koff_h[s]:koff_h[s + 1]])
        ref = oracle.pack(oracle.bank_session(s, np_view(b.keys[lo:hi]), np_view(b.values[lo:hi]),
                                              kp, kdt, vdt))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), s
        refs.append((kp, lo, hi))
    # Excursion: the live banks are overwritten; restore compacted banks.
    for t in keys + vals:
        t.zero_()
    outs, tg = [], []
    for s in range(b.sessions):
        k = ks[s]
        o = (torch.full((k,), -1, dtype=torch.int32, device=dev),
             torch.zeros((k,) + tuple(b.keys.shape[1:]), dtype=b.keys.dtype, device=dev),
             torch.zeros((k,) + tuple(b.values.shape[1:]), dtype=b.values.dtype, device=dev))
        outs.append(o)
        tg.append(pcs.bank_targets(s, *o))
    ctx.restore(snaps, tg, verify=True)
    torch.cuda.synchronize()
    for s, (kp, lo, hi) in enumerate(refs):
        oi, ok, ov = outs[s]
        assert oi.cpu().numpy().tolist() == kp.tolist()
        assert torch.equal(ok.cpu(), b.keys[lo:hi][kp]), s
        assert torch.equal(ov.cpu(), b.values[lo:hi][kp]), s
    for sn in snaps:
        ctx.delete(sn)


def test_bank_config2_full(ctx, dev):
    # 64 sessions, n ~ U[1,512], fp16[256] keys, bf16[16,32,32] latents, k = min(n,128).
    b = synth.banks_config2()
    _bank_round_trip(ctx, b, dev, ctx.params(pcs.PCS_K_FIXED, k_max=128), pcs.PCS_PLACE_DEVICE)


def test_bank_budget_to_pinned_host(ctx, dev):
    # Config 5's shape at a reduced session count: budget rule, pinned host.
    b = synth.banks_config5(sessions=24, n_lo=256, n_hi=1024)
    E = 1024 + 2048
    B = sum(b.n) * E * 5 // 8
    _bank_round_trip(ctx, b, dev, ctx.params(pcs.PCS_K_BUDGET, budget=B),
                     pcs.PCS_PLACE_PINNED_HOST)


# ---------------------------------------------------------------------------
# Windowed paged KV (config 3 shape, reduced)
# ---------------------------------------------------------------------------

def _kv_logical(pool, pt, start, window, page_rows):
    j = torch.arange(window)
    slot = (start + j) % window
    return pool[pt.long()[slot // page_rows], slot % page_rows]


@pytest.mark.parametrize("starts", [[0, 15, 16, 1023], [1, 512, 1000, 17]])
def test_kv_pack_restore_fresh_pool(ctx, dev, starts):
    kv = synth.kv(seed=33, sessions=4, layers=3, heads=4, head_dim=64, window=1024, page_rows=16)
    kp_h, vp_h = kv.k_pool.clone(), kv.v_pool.clone()
    kp, vp = kv.k_pool.to(dev), kv.v_pool.to(dev)
    pt = kv.page_table.to(dev)
    meta = kv.meta.to(dev)
    sess = [pcs.kv_session(s, meta[s], kp, vp, pt[s], starts[s], kv.window)
            for s in range(kv.sessions)]
    snaps = ctx.checkpoint(sess)
    for s in range(kv.sessions):
        ref = oracle.pack(oracle.kv_session(s, kv.meta[s].numpy(), np_view(kp_h), np_view(vp_h),
                                            kv.page_table[s].numpy(), starts[s], kv.window,
                                            kv.page_rows, kv.row_bytes))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), s
    # Restore into a freshly permuted, zeroed pool at the stored ring starts.
    pt2 = synth.page_permutation(99, kv.sessions, kv.layers, kv.window // kv.page_rows).to(dev)
    kp2, vp2 = torch.zeros_like(kp), torch.zeros_like(vp)
    meta2 = torch.zeros_like(meta)
    tg = [pcs.kv_session(s, meta2[s], kp2, vp2, pt2[s], pcs.PCS_RING_START_FROM_SNAPSHOT,
                         kv.window) for s in range(kv.sessions)]
    ctx.restore(snaps, tg, verify=True)
    torch.cuda.synchronize()
    assert torch.equal(meta2.cpu(), kv.meta)
    pt2h = pt2.cpu()
    for s in range(kv.sessions):
        for l in range(kv.layers):
            a = _kv_logical(kp2.cpu(), pt2h[s, l], starts[s], kv.window, kv.page_rows)
            b = _kv_logical(kp_h, kv.page_table[s, l], starts[s], kv.window, kv.page_rows)
            assert torch.equal(a, b), (s, l)
            a = _kv_logical(vp2.cpu(), pt2h[s, l], starts[s], kv.window, kv.page_rows)
            b = _kv_logical(vp_h, kv.page_table[s, l], starts[s], kv.window, kv.page_rows)
            assert torch.equal(a, b), (s, l)
    for sn in snaps:
        ctx.delete(sn)


def test_kv_odd_geometry(ctx, dev):
    # Page size and row size not powers of two (division path), window 96.
    kv = synth.kv(seed=34, sessions=2, layers=2, heads=3, head_dim=8, window=96, page_rows=12)
    kp, vp, pt, meta = kv.k_pool.to(dev), kv.v_pool.to(dev), kv.page_table.to(dev), kv.meta.to(dev)
    for start in [0, 11, 12, 95]:
        snap = ctx.checkpoint([pcs.kv_session(0, meta[0], kp, vp, pt[0], start, kv.window)])[0]
        ref = oracle.pack(oracle.kv_session(0, kv.meta[0].numpy(), np_view(kv.k_pool),
                                            np_view(kv.v_pool), kv.page_table[0].numpy(), start,
                                            kv.window, kv.page_rows, kv.row_bytes))
        assert np.array_equal(ctx.record(snap).numpy(), ref), start
        ctx.delete(snap)


# ---------------------------------------------------------------------------
# Fork, durability, error paths
# ---------------------------------------------------------------------------

def test_fork_independence(ctx, dev):
    m = synth.markov(seed=41)
    obs, rng = m.obs.to(dev), m.rng.to(dev)
    parent = ctx.checkpoint([pcs.markov_session(1, obs, rng)])[0]
    pref = ctx.record(parent).numpy().copy()
    child = ctx.fork(parent)
    assert np.array_equal(ctx.record(child).numpy(), pref)
    # Restore the child, diverge, re-checkpoint: the parent is untouched (I3).
    ctx.restore([child], [pcs.markov_session(1, obs, rng)])
    obs[0, 0, :10] ^= 0x55
    ctx.delete(child)
    child2 = ctx.checkpoint([pcs.markov_session(1, obs, rng)])[0]
    assert ctx.info(child2).session_fp != ctx.info(parent).session_fp
    assert np.array_equal(ctx.record(parent).numpy(), pref)
    ctx.delete(child2)
    ctx.delete(parent)


def test_file_round_trip_and_corruption(ctx, dev, tmp_path):
    m = synth.markov(seed=42)
    obs, rng = m.obs.to(dev), m.rng.to(dev)
    snap = ctx.checkpoint([pcs.markov_session(5, obs, rng)])[0]
    ref = ctx.record(snap).numpy().copy()
    path = str(tmp_path / "s.pcs")
    ctx.write_file(snap, path)
    assert np.array_equal(np.fromfile(path, dtype=np.uint8), ref)
    for place in [pcs.PCS_PLACE_DEVICE, pcs.PCS_PLACE_PINNED_HOST]:
        back = ctx.read_file(path, place)
        assert np.array_equal(ctx.record(back).numpy(), ref)
        o, r = torch.zeros_like(obs), torch.zeros_like(rng)
        ctx.restore([back], [pcs.markov_session(5, o, r)], verify=True)
        torch.cuda.synchronize()
        assert torch.equal(o, obs) and torch.equal(r, rng)
        ctx.delete(back)
    # A flipped payload byte is caught by verification.
    bad = ref.copy()
    bad[ctx.section(snap, 0).offset + 1000] ^= 4
    bad.tofile(path)
    back = ctx.read_file(path)
    o, r = torch.zeros_like(obs), torch.zeros_like(rng)
    st = ctx.restore_status([back], [pcs.markov_session(5, o, r)], verify=True)
    assert st == pcs.PCS_E_CORRUPT
    ctx.delete(back)
    # Malformed headers are refused at read time.
    for mutate in [lambda a: a.__setitem__(0, a[0] ^ 1),           # magic
                   lambda a: a.__setitem__(64 + 16, 3)]:            # section offset
        bad = ref.copy()
        mutate(bad)
        bad.tofile(path)
        with pytest.raises(pcs.PcsError) as e:
            ctx.read_file(path)
        assert e.value.status == pcs.PCS_E_CORRUPT
    ref[:100].tofile(path)
    with pytest.raises(pcs.PcsError):
        ctx.read_file(path)
    ctx.delete(snap)


def test_bad_handle_and_shape_errors(ctx, dev):
    m = synth.markov(seed=43, shape=(3, 8, 8))
    obs, rng = m.obs.to(dev), m.rng.to(dev)
    snap = ctx.checkpoint([pcs.markov_session(1, obs, rng)])[0]
    with pytest.raises(pcs.PcsError) as e:
        ctx.restore([snap], [pcs.markov_session(1, obs.reshape(-1)[:100], rng)])
    assert e.value.status == pcs.PCS_E_INVAL
    handle = snap.handle
    ctx.delete(snap)
    snap.handle = handle
    with pytest.raises(pcs.PcsError) as e:
        ctx.info(snap)
    assert e.value.status == pcs.PCS_E_HANDLE


def test_index_out_of_range_is_reported_not_accessed(ctx, dev):
    keys = torch.randn(10, 64, device=dev).half()
    vals = torch.zeros(10, 32, dtype=torch.uint8, device=dev)
    kept = torch.tensor([0, 3, 10 + 5], dtype=torch.int32, device=dev)
    snap = ctx.checkpoint([pcs.bank_session(0, keys, vals, kept)])[0]
    with pytest.raises(pcs.PcsError) as e:
        ctx.sync()
    assert e.value.status == pcs.PCS_E_RANGE
    ctx.sync()  # cleared
    ctx.delete(snap)


def test_mixed_kinds_one_call(ctx, dev):
    m = synth.markov(seed=50, shape=(3, 40, 40))
    kv = synth.kv(seed=51, sessions=1, layers=2, heads=2, head_dim=64, window=64, page_rows=16)
    b = synth.banks(52, 1, 30, 30, 64, torch.bfloat16, (128,), torch.uint8)
    kept = torch.arange(0, 30, 3, dtype=torch.int32)
    sess = [pcs.markov_session(0, m.obs.to(dev), m.rng.to(dev)),
            pcs.kv_session(1, kv.meta[0].to(dev), kv.k_pool.to(dev), kv.v_pool.to(dev),
                           kv.page_table[0].to(dev), 7, kv.window),
            pcs.bank_session(2, b.keys.to(dev), b.values.to(dev), kept.to(dev))]
    snaps = ctx.checkpoint(sess)
    refs = [oracle.pack(oracle.markov_session(0, m.obs.numpy(), m.rng.numpy().view(np.uint64))),
            oracle.pack(oracle.kv_session(1, kv.meta[0].numpy(), np_view(kv.k_pool),
                                          np_view(kv.v_pool), kv.page_table[0].numpy(), 7,
                                          kv.window, kv.page_rows, kv.row_bytes)),
            oracle.pack(oracle.bank_session(2, np_view(b.keys), np_view(b.values), kept.numpy(),
                                            oracle.DT_BF16, oracle.DT_U8))]
    for s, r in zip(snaps, refs):
        assert np.array_equal(ctx.record(s).numpy(), r)
        ctx.delete(s)


@pytest.mark.parametrize("D,dtype", [(8, torch.float16), (264, torch.bfloat16),
                                     (1024, torch.float16), (1536, torch.bfloat16)])
def test_prune_key_dims(ctx, dev, D, dtype):
    # Every code path of the score kernel: 1, 2, 4 segments per lane and the
    # generic loop for D > 1024.
    b = synth.banks(70 + D, 9, 1, 70, D, dtype, (8,), torch.uint8)
    keys, vals, qs = _bank_views(b, dev)
    _check_prune(ctx, b, keys, qs, ctx.params(pcs.PCS_K_FRACTION, fraction=0.3), dev)


def test_async_verify_and_batch_forms(ctx, dev, tmp_path):
    # verify = 2 checks on the device and reports at the next pcs_sync.
    ms = [synth.markov(seed=300 + i, shape=(3, 20, 20)) for i in range(5)]
    sess = [pcs.markov_session(i, m.obs.to(dev), m.rng.to(dev)) for i, m in enumerate(ms)]
    arr = ctx.session_array(sess)
    hs = ctx.checkpoint_raw(arr, 5)
    outs = [pcs.markov_session(i, torch.zeros_like(m.obs, device=dev),
                               torch.zeros_like(m.rng, device=dev)) for i, m in enumerate(ms)]
    oarr = ctx.session_array(outs)
    ctx.restore_raw(hs, 5, oarr, verify=2)
    ctx.sync()
    for m, o in zip(ms, outs):
        assert torch.equal(o.keep[0].cpu(), m.obs) and torch.equal(o.keep[1].cpu(), m.rng)
    # A corrupted record read from a file: no error at restore, one at sync.
    snap = pcs.Snapshot(ctx, hs[2])
    path = str(tmp_path / "c.pcs")
    ctx.write_file(snap, path)
    raw = np.fromfile(path, dtype=np.uint8)
    raw[ctx.section(snap, 0).offset + 5] ^= 0x20
    raw.tofile(path)
    bad = ctx.read_file(path)
    ctx.restore([bad], [outs[2]], verify=2)
    with pytest.raises(pcs.PcsError) as e:
        ctx.sync()
    assert e.value.status == pcs.PCS_E_CORRUPT
    ctx.sync()  # cleared
    ctx.delete(bad)
    # delete_many: all or nothing.
    import ctypes
    junk = (ctypes.c_void_p * 2)(hs[0], 12345)
    with pytest.raises(pcs.PcsError) as e:
        ctx.delete_raw(junk, 2)
    assert e.value.status == pcs.PCS_E_HANDLE
    assert ctx.stats().live_snapshots >= 5
    ctx.delete_raw(hs, 5)
    with pytest.raises(pcs.PcsError):
        ctx.delete_raw(hs, 1)


def test_prune_mixed_key_types(ctx, dev):
    # fp16 and bf16 banks in one call take the general score kernel.
    b1 = synth.banks(80, 3, 5, 60, 128, torch.float16, (8,), torch.uint8)
    b2 = synth.banks(81, 3, 5, 60, 128, torch.bfloat16, (8,), torch.uint8)
    keys = [x.to(dev) for x in _bank_views(b1, "cpu")[0] + _bank_views(b2, "cpu")[0]]
    qs = [x.to(dev) for x in _bank_views(b1, "cpu")[2] + _bank_views(b2, "cpu")[2]]
    banks = ctx.banks_array(keys, qs, 272)
    p = ctx.params(pcs.PCS_K_FIXED, k_max=7)
    ks = ctx.prune_counts(banks, 6, p)
    kept = torch.empty(sum(ks), dtype=torch.int32, device=dev)
    scores = torch.empty(sum(k.shape[0] for k in keys), dtype=torch.float32, device=dev)
    ctx.prune(banks, 6, p, kept, None, scores)
    ctx.sync()
    sc, kh = scores.cpu().numpy(), kept.cpu().numpy()
    off = eo = 0
    for k, q, kk in zip(keys, qs, ks):
        s32 = oracle.scores(np_view(q), np_view(k))
        n = k.shape[0]
        assert np.array_equal(sc[eo:eo + n].view(np.uint32), s32.view(np.uint32))
        assert kh[off:off + kk].tolist() == oracle.topk(s32, kk).tolist()
        off += kk
        eo += n


@pytest.mark.parametrize("policy", ["lru", "fifo"])
def test_topk_by_recency_keys(ctx, dev, policy):
    # Recency-keyed retention (Table tab:evict lru / fifo): rank keys supplied
    # by the caller; ties by entry index.
    rnd = np.random.default_rng(7)
    n = rnd.integers(1, 300, 20).tolist()
    k = [max(1, int(x * 0.12 + 0.5)) for x in n]
    if policy == "lru":
        keys = [rnd.integers(0, 50, x).astype(np.float32) for x in n]  # last-use step (ties)
    else:
        keys = [np.arange(x, dtype=np.float32) for x in n]             # insertion order
    flat = torch.from_numpy(np.concatenate(keys)).to(dev)
    kept = torch.empty(sum(min(a, b) for a, b in zip(n, k)), dtype=torch.int32, device=dev)
    koff = torch.empty(len(n) + 1, dtype=torch.int32, device=dev)
    ctx.topk(flat, n, k, kept, koff)
    ctx.sync()
    kh, oh = kept.cpu().numpy(), koff.cpu().numpy()
    for b, (kk, x) in enumerate(zip(keys, k)):
        assert kh[oh[b]:oh[b + 1]].tolist() == oracle.topk(kk, x).tolist(), b
    if policy == "fifo":
        assert kh[oh[0]:oh[1]].tolist() == list(range(n[0] - k[0], n[0]))


@pytest.mark.parametrize("ties", [False, True])
def test_topk_bank_sizes(ctx, dev, ties):
    # Banks up to 4096 entries are selected from registers, larger ones by
    # re-reading their keys: sizes on both sides of the switch, several k.
    rnd = np.random.default_rng(17 + ties)
    n = [1, 17, 255, 256, 257, 4095, 4096, 4097, 10000, 3000]
    k = [1, 5, 1, 128, 256, 4094, 1000, 4096, 3333, 2999]
    if ties:
        keys = [rnd.integers(0, 40, x).astype(np.float32) for x in n]
    else:
        keys = [rnd.normal(size=x).astype(np.float32) for x in n]
    keys[3][:] = 0.0  # one bank of equal keys
    flat = torch.from_numpy(np.concatenate(keys)).to(dev)
    kept = torch.empty(sum(k), dtype=torch.int32, device=dev)
    koff = torch.empty(len(n) + 1, dtype=torch.int32, device=dev)
    ctx.topk(flat, n, k, kept, koff)
    ctx.sync()
    kh, oh = kept.cpu().numpy(), koff.cpu().numpy()
    for b, (kk, x) in enumerate(zip(keys, k)):
        assert kh[oh[b]:oh[b + 1]].tolist() == oracle.topk(kk, x).tolist(), b


def test_topk_digit_boundaries(ctx, dev):
    # Keys that share their leading bits and differ only in the last digit,
    # keys straddling digit boundaries, special values (NaN lowest, -0 == +0,
    # infinities, subnormals) and runs of equal keys at the threshold.
    rnd = np.random.default_rng(29)
    banks = []
    one = np.float32(1.0).view(np.uint32)
    banks.append((one + rnd.integers(0, 1024, 3000)).astype(np.uint32).view(np.float32))
    banks.append((one + rnd.integers(0, 1 << 21, 2048)).astype(np.uint32).view(np.float32))
    spec = np.array([np.nan, 0.0, -0.0, np.inf, -np.inf, 1e-45, -1e-45, 1e-38, -2.5, 2.5],
                    dtype=np.float32)
    banks.append(rnd.choice(spec, 1500))
    eq = rnd.normal(size=4096).astype(np.float32)
    eq[rnd.integers(0, 4096, 1500)] = np.float32(0.125)
    banks.append(eq)
    banks.append(-np.abs(rnd.normal(size=700)).astype(np.float32))
    k = [1500, 1024, 700, 2000, 350]
    flat = torch.from_numpy(np.concatenate(banks)).to(dev)
    n = [len(x) for x in banks]
    kept = torch.empty(sum(k), dtype=torch.int32, device=dev)
    koff = torch.empty(len(n) + 1, dtype=torch.int32, device=dev)
    ctx.topk(flat, n, k, kept, koff)
    ctx.sync()
    kh, oh = kept.cpu().numpy(), koff.cpu().numpy()
    for b, (kk, x) in enumerate(zip(banks, k)):
        assert kh[oh[b]:oh[b + 1]].tolist() == oracle.topk(kk, x).tolist(), b


def test_fork_many_mixed_placements(ctx, dev):
    # Device records over 1 MiB take the TMA copy; pinned-host ones the register copy.
    kv = synth.kv(seed=90, sessions=3, layers=2, heads=16, head_dim=64, window=256, page_rows=16)
    kp, vp, pt, meta = kv.k_pool.to(dev), kv.v_pool.to(dev), kv.page_table.to(dev), kv.meta.to(dev)
    sess = [pcs.kv_session(s, meta[s], kp, vp, pt[s], kv.ring_start[s], kv.window) for s in range(3)]
    dev_snaps = ctx.checkpoint(sess)
    host_snaps = ctx.checkpoint(sess, placement=pcs.PCS_PLACE_PINNED_HOST)
    import ctypes
    parents = dev_snaps + host_snaps
    hs = (ctypes.c_void_p * 6)(*[x.handle for x in parents])
    kids = ctx.fork_raw(hs, 6)
    for i, p in enumerate(parents):
        child = pcs.Snapshot(ctx, kids[i])
        assert ctx.info(child).placement == ctx.info(p).placement
        assert np.array_equal(ctx.record(child).numpy(), ctx.record(p).numpy()), i
    ctx.delete_raw(kids, 6)
    for x in parents:
        ctx.delete(x)


def test_prune_kept_align_16_bytes(ctx, dev):
    """kept_align = 4: each bank's kept list starts at a multiple of four
    entries; the lists are the oracle's top-k, kept_off gives the padded
    offsets, and a checkpoint of the banks equals the oracle's records."""
    b = synth.banks_config2(seed=91, sessions=12)
    keys, vals, qs = _bank_views(b, dev)
    banks = ctx.banks_array(keys, qs, 512 + b.value_bytes)
    for bad in (2, 3, 8):
        with pytest.raises(pcs.PcsError) as e:
            ctx.prune(banks, b.sessions, ctx.params(pcs.PCS_K_FIXED, k_max=7, kept_align=bad),
                      torch.empty(1024, dtype=torch.int32, device=dev))
        assert e.value.status == pcs.PCS_E_INVAL
    params = ctx.params(pcs.PCS_K_FIXED, k_max=37, kept_align=4)
    ks = ctx.prune_counts(banks, b.sessions, params)
    off = np.concatenate([[0], np.cumsum([(k + 3) // 4 * 4 for k in ks])]).astype(np.int64)
    kept = torch.full((int(off[-1]),), -7, dtype=torch.int32, device=dev)
    koff = torch.empty(b.sessions + 1, dtype=torch.int32, device=dev)
    ctx.prune(banks, b.sessions, params, kept, koff)
    assert koff.cpu().numpy().tolist() == off.tolist()
    kept_h = kept.cpu().numpy()
    for s in range(b.sessions):
        sc = oracle.scores(np_view(b.queries[s]), np_view(keys[s].cpu()))
        assert kept_h[off[s]:off[s] + ks[s]].tolist() == oracle.topk(sc, 37).tolist(), s
        assert (kept_h[off[s] + ks[s]:off[s + 1]] == -7).all()  # padding untouched
    sess = [pcs.bank_session(s, keys[s], vals[s], kept[int(off[s]):int(off[s]) + ks[s]])
            for s in range(b.sessions)]
    snaps = ctx.checkpoint(sess)
    kdt = oracle.DT_F16 if b.keys.dtype == torch.float16 else oracle.DT_BF16
    vdt = oracle.DT_BF16 if b.values.dtype == torch.bfloat16 else oracle.DT_U8
    for s in range(b.sessions):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        ref = oracle.pack(oracle.bank_session(s, np_view(b.keys[lo:hi]), np_view(b.values[lo:hi]),
                                              np.ascontiguousarray(kept_h[off[s]:off[s] + ks[s]]),
                                              kdt, vdt))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), s
        ctx.delete(snaps[s])
