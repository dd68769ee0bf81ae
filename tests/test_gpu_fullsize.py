"""GPU parity at the full workload sizes, in the launch shape bench.py times.

Every fingerprint the GPU stores or returns at full size is compared with
the oracle's: the oracle's C calls release the GIL, so host threads (one per
core) fingerprint the records' payloads side by side.  Whole records are
compared byte for byte with the oracle's on sampled sessions (its pack would
re-gather every page on the host), and every payload byte of every record is
compared on the device with a gather of the source rows in logical order.
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_view

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def _session_pages(pool, pt):
    """The pages a session uses, compacted, with the page table renumbered."""
    flat = pt.reshape(-1).long()
    pages = pool[flat].cpu()
    return pages, torch.arange(flat.numel(), dtype=torch.int32).view(pt.shape)


def _host_threads() -> int:
    return max(1, len(os.sched_getaffinity(0)))


def _check_record_fps(ctx, snaps, batch=32):
    """Every section fp and the session fp of every record against the
    oracle: fp of each payload as the record holds it, and the session fp
    composed from the oracle's section fps by the oracle's tree and mixer."""
    sizes = [ctx.info(x).total_bytes for x in snaps]
    stage = torch.empty(max(sizes) * min(batch, len(snaps)), dtype=torch.uint8, pin_memory=True)
    host = stage.numpy()
    checked = 0
    with ThreadPoolExecutor(_host_threads()) as pool:
        for b0 in range(0, len(snaps), batch):
            group = snaps[b0:b0 + batch]
            offs = np.cumsum([0] + sizes[b0:b0 + len(group)]).tolist()
            for i, x in enumerate(group):
                ctx.copy_out(x, 0, sizes[b0 + i], stage[offs[i]:offs[i + 1]])
            torch.cuda.current_stream().synchronize()
            jobs = []
            for i, x in enumerate(group):
                info = ctx.info(x)
                secs = [ctx.section(x, j) for j in range(info.n_sections)]
                futs = [pool.submit(oracle.fingerprint,
                                    host[offs[i] + e.offset: offs[i] + e.offset + e.bytes])
                        for e in secs]
                jobs.append((b0 + i, info, secs, futs))
            for s, info, secs, futs in jobs:
                fps = [f.result() for f in futs]
                assert [e.fp for e in secs] == fps, s
                assert info.session_fp == oracle.fmix(oracle.tree(fps) ^ info.n_sections), s
                checked += 1
    assert checked == len(snaps)


def test_kv_full_size(ctx, dev):
    # 256 sessions x 24 layers x 16 heads x 64, window 1024, 16-token pages.
    kv = synth.kv(device=dev)
    S, Lyr, W, P = kv.sessions, kv.layers, kv.window, kv.page_rows
    sess = [pcs.kv_session(s, kv.meta[s], kv.k_pool, kv.v_pool, kv.page_table[s], kv.ring_start[s], W)
            for s in range(S)]
    snaps = ctx.checkpoint(sess)
    pt2 = synth.page_permutation(synth.seed_for(3) + 7, S, Lyr, W // P, device=dev)
    k2, v2 = torch.empty_like(kv.k_pool), torch.empty_like(kv.v_pool)
    meta2 = torch.empty_like(kv.meta)
    tg = [pcs.kv_session(s, meta2[s], k2, v2, pt2[s], pcs.PCS_RING_START_FROM_SNAPSHOT, W)
          for s in range(S)]
    ctx.restore(snaps, tg, verify=True)
    torch.cuda.synchronize()
    # Every restored row of every session equals its source row.
    j = torch.arange(W, device=dev)
    for s in range(S):
        slot = (kv.ring_start[s] + j) % W
        a = kv.page_table[s].long()[:, slot // P]
        b = pt2[s].long()[:, slot // P]
        r = slot % P
        assert torch.equal(kv.k_pool[a, r], k2[b, r]), s
        assert torch.equal(kv.v_pool[a, r], v2[b, r]), s
    assert torch.equal(meta2, kv.meta)
    # Every payload byte of every record: META, then K_l and V_l of every
    # layer in logical order (token j = ring slot (start + j) mod window).
    layer_bytes = W * kv.k_pool[0, 0].numel() * 2
    rec = torch.empty(ctx.info(snaps[0]).total_bytes, dtype=torch.uint8, device=dev)
    for s in range(S):
        ctx.copy_out(snaps[s], 0, rec.numel(), rec)
        slot = (kv.ring_start[s] + j) % W
        e0 = ctx.section(snaps[s], 0)
        assert torch.equal(rec[e0.offset:e0.offset + e0.bytes], kv.meta[s].view(torch.uint8)), s
        for l in range(Lyr):
            rows = slot // P
            for i, pool in ((1 + 2 * l, kv.k_pool), (2 + 2 * l, kv.v_pool)):
                e = ctx.section(snaps[s], i)
                assert e.bytes == layer_bytes
                want = pool[kv.page_table[s, l].long()[rows], slot % P].contiguous()
                assert torch.equal(rec[e.offset:e.offset + e.bytes], want.view(-1).view(torch.uint8)), (s, l, i)
    # Every section fp and session fp of every record against the oracle.
    _check_record_fps(ctx, snaps)
    # Sampled whole records against the oracle.
    for s in (0, 127, S - 1):
        kp, ptc = _session_pages(kv.k_pool, kv.page_table[s])
        vp, _ = _session_pages(kv.v_pool, kv.page_table[s])
        ref = oracle.pack(oracle.kv_session(s, kv.meta[s].cpu().numpy(), np_view(kp), np_view(vp),
                                            ptc.numpy(), kv.ring_start[s], W, P, kv.row_bytes))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), s
    for x in snaps:
        ctx.delete(x)


def test_mass_banks_full_size(ctx, dev):
    # 2048 sessions, n ~ U[256,4096], key bf16[512], value u8[2048], query
    # bf16[512]; host budget 8 GiB; pack to pinned host, restore to HBM.
    b = synth.banks_config5(device=dev)
    S = b.sessions
    E = 1024 + 2048
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    vals = [b.values[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    qs = [b.queries[s] for s in range(S)]
    banks = ctx.banks_array(keys, qs, E)
    params = ctx.params(pcs.PCS_K_BUDGET, budget=8 << 30)
    ks = ctx.prune_counts(banks, S, params)
    assert sum(ks) * E <= 8 << 30
    kept = torch.empty(sum(ks), dtype=torch.int32, device=dev)
    koff = torch.empty(S + 1, dtype=torch.int32, device=dev)
    scores = torch.empty(b.keys.shape[0], dtype=torch.float32, device=dev)
    ctx.prune(banks, S, params, kept, koff, scores)
    koff_h = koff.cpu().tolist()
    sess = [pcs.bank_session(s, keys[s], vals[s], kept[koff_h[s]:koff_h[s + 1]]) for s in range(S)]
    snaps = ctx.checkpoint(sess, placement=pcs.PCS_PLACE_PINNED_HOST)
    outs = [(torch.empty(ks[s], dtype=torch.int32, device=dev),
             torch.empty(ks[s], 512, dtype=torch.bfloat16, device=dev),
             torch.empty(ks[s], 2048, dtype=torch.uint8, device=dev)) for s in range(S)]
    ctx.restore(snaps, [pcs.bank_targets(s, *outs[s]) for s in range(S)], verify=True)
    torch.cuda.synchronize()
    # Every restored bank equals the kept rows of the live bank.
    for s in range(S):
        ki = kept[koff_h[s]:koff_h[s + 1]]
        assert torch.equal(outs[s][0], ki), s
        assert torch.equal(outs[s][1], keys[s][ki.long()]), s
        assert torch.equal(outs[s][2], vals[s][ki.long()]), s
        assert bool((ki[1:] > ki[:-1]).all()), s
    # Sampled banks against the oracle: scores (bit-exact fp32, 1e-3 vs fp64),
    # kept sets, whole records.
    sc = scores.cpu().numpy()
    kept_h = kept.cpu().numpy()
    for s in (0, 1, 1000, S - 1):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        kh, vh = np_view(keys[s]), vals[s].cpu().numpy()
        s32, s64 = oracle.scores(np_view(qs[s]), kh, want64=True)
        assert np.array_equal(sc[lo:hi].view(np.uint32), s32.view(np.uint32)), s
        np.testing.assert_allclose(sc[lo:hi], s64, rtol=1e-3, atol=1e-6)
        want = oracle.topk(s32, ks[s])
        assert kept_h[koff_h[s]:koff_h[s + 1]].tolist() == want.tolist(), s
        ref = oracle.pack(oracle.bank_session(s, kh, vh, want, oracle.DT_BF16, oracle.DT_U8))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), s
    for x in snaps:
        ctx.delete(x)


def _ord32_np(s):
    u = s.view(np.uint32).astype(np.uint64)
    out = np.where(u & 0x80000000, (~u) & 0xFFFFFFFF, u | 0x80000000)
    out[s == 0] = 0x80000000
    out[np.isnan(s)] = 0
    return out


def test_global_threshold_full_size(ctx, dev):
    # The same 2048 banks under one relevance threshold across all of them:
    # sampled scores against the oracle, then the defining property at full
    # size -- the kept set is the longest prefix of the (score desc, bank,
    # index) order whose bytes fit 8 GiB.
    b = synth.banks_config5(device=dev)
    S, E, B = b.sessions, 1024 + 2048, 8 << 30
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    qs = [b.queries[s] for s in range(S)]
    banks = ctx.banks_array(keys, qs, E)
    total = b.keys.shape[0]
    kept = torch.empty(total, dtype=torch.int32, device=dev)
    koff = torch.empty(S + 1, dtype=torch.int32, device=dev)
    scores = torch.empty(total, dtype=torch.float32, device=dev)
    ctx.prune_global(banks, S, B, kept, koff, scores)
    sc = scores.cpu().numpy()
    koff_h = koff.cpu().numpy().astype(np.int64)
    kept_h = kept.cpu().numpy()[:koff_h[-1]]
    for s in (0, 777, S - 1):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        s32 = oracle.scores(np_view(qs[s]), np_view(keys[s]))
        assert np.array_equal(sc[lo:hi].view(np.uint32), s32.view(np.uint32)), s
    m = min(B // E, total)
    assert koff_h[-1] == m and koff_h[0] == 0 and np.all(np.diff(koff_h) >= 0)
    pos = np.arange(total, dtype=np.uint64)
    key = (_ord32_np(sc) << np.uint64(32)) | (np.uint64(0xFFFFFFFF) - pos)
    top = np.sort(np.argsort(key)[::-1][:m])
    starts = np.asarray(b.entry_off[:-1], dtype=np.int64)
    got = np.concatenate([starts[s] + kept_h[koff_h[s]:koff_h[s + 1]] for s in range(S)])
    assert np.array_equal(got, top)


def test_markov_batch_full_size(ctx, dev):
    # 4096 Markovian sessions of [3,256,256] uint8 + 16-byte RNG in one call.
    S = 4096
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(1))
    obs = torch.randint(0, 256, (S, 3, 256, 256), generator=g, device=dev, dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (S, 2), generator=g, device=dev, dtype=torch.int64)
    sess = [pcs.markov_session(s, obs[s], rng[s]) for s in range(S)]
    snaps = ctx.checkpoint(sess)
    o2, r2 = torch.zeros_like(obs), torch.zeros_like(rng)
    ctx.restore(snaps, [pcs.markov_session(s, o2[s], r2[s]) for s in range(S)], verify=True)
    torch.cuda.synchronize()
    assert torch.equal(o2, obs) and torch.equal(r2, rng)
    for s in (0, S // 2, S - 1):
        ref = oracle.pack(oracle.markov_session(s, obs[s].cpu().numpy(),
                                                rng[s].cpu().numpy().view(np.uint64)))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), s
    for x in snaps:
        ctx.delete(x)
