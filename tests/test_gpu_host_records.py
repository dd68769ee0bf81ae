"""GPU parity: records in pinned host memory.

Records in pinned host memory are the paper's resting place of a suspended
session's PCS (Sec. 5 "Structure").  The library's register kernel writes
and reads them over the host link, on half the SMs (a call that only crosses
the link).  A checkpoint's host records equal the oracle's byte for byte, a
verified restore from them brings back every byte (I1) and reports a
corrupted record (PCS_E_CORRUPT), and prepared calls track the sessions'
current bytes.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth

pytestmark = pytest.mark.gpu


def _markov(n, dev, seed):
    g = torch.Generator(device=dev).manual_seed(seed)
    obs = torch.randint(0, 256, (n, 3, 256, 256), generator=g, device=dev, dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (n, 2), generator=g, device=dev, dtype=torch.int64)
    return obs, rng


def _oracle_markov(s, obs, rng):
    return oracle.pack(oracle.markov_session(s, obs[s].cpu().numpy(),
                                             rng[s].cpu().numpy().view(np.uint64)))


def _timed(ctx, fn):
    ctx.timing(True)
    out = fn()
    torch.cuda.synchronize()
    t = ctx.kernel_times()
    ctx.timing(False)
    return out, t


def test_host_records_and_restore(ctx, dev):
    n = 8  # 1.6 MB: past the fused small-call path
    obs, rng = _markov(n, dev, 900)
    sess = [pcs.markov_session(s, obs[s], rng[s]) for s in range(n)]
    snaps, t = _timed(ctx, lambda: ctx.checkpoint(sess, placement=pcs.PCS_PLACE_PINNED_HOST))
    assert "k_stream<pack>" in t and "k_bulk<pack>" not in t
    for s in range(n):
        assert ctx.info(snaps[s]).placement == pcs.PCS_PLACE_PINNED_HOST
        assert np.array_equal(ctx.record(snaps[s]).numpy(), _oracle_markov(s, obs, rng)), s
    o2, r2 = torch.zeros_like(obs), torch.zeros_like(rng)
    tg = [pcs.markov_session(s, o2[s], r2[s]) for s in range(n)]
    _, t = _timed(ctx, lambda: ctx.restore(snaps, tg, verify=True))
    assert "k_stream<restore_verify>" in t and "k_bulk<restore_verify>" not in t
    assert torch.equal(o2, obs) and torch.equal(r2, rng)
    # Every other snapshot: records that are not adjacent in host memory.
    o3, r3 = torch.zeros_like(obs), torch.zeros_like(rng)
    pick = list(range(0, n, 2))
    ctx.restore([snaps[s] for s in pick], [pcs.markov_session(s, o3[s], r3[s]) for s in pick],
                verify=True)
    torch.cuda.synchronize()
    for s in range(n):
        want = (obs[s], rng[s]) if s % 2 == 0 else (torch.zeros_like(obs[s]), torch.zeros_like(rng[s]))
        assert torch.equal(o3[s], want[0]) and torch.equal(r3[s], want[1]), s
    for x in snaps:
        ctx.delete(x)


def test_host_kv_records(ctx, dev):
    kv = synth.kv(seed=77, sessions=3, layers=2, heads=4, head_dim=64, window=256, page_rows=16,
                  device=dev)
    W, P = kv.window, kv.page_rows
    sess = [pcs.kv_session(s, kv.meta[s], kv.k_pool, kv.v_pool, kv.page_table[s], kv.ring_start[s], W)
            for s in range(kv.sessions)]
    snaps = ctx.checkpoint(sess, placement=pcs.PCS_PLACE_PINNED_HOST)
    for s in range(kv.sessions):
        flat = kv.page_table[s].reshape(-1).long()
        ptc = torch.arange(flat.numel(), dtype=torch.int32).view(kv.page_table[s].shape)
        kp = kv.k_pool[flat].cpu().view(torch.int16).numpy().view(np.uint16)
        vp = kv.v_pool[flat].cpu().view(torch.int16).numpy().view(np.uint16)
        ref = oracle.pack(oracle.kv_session(s, kv.meta[s].cpu().numpy(), kp, vp, ptc.numpy(),
                                            kv.ring_start[s], W, P, kv.row_bytes))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), s
    pt2 = synth.page_permutation(78, kv.sessions, kv.layers, W // P, device=dev)
    k2, v2, m2 = torch.zeros_like(kv.k_pool), torch.zeros_like(kv.v_pool), torch.zeros_like(kv.meta)
    ctx.restore(snaps, [pcs.kv_session(s, m2[s], k2, v2, pt2[s], pcs.PCS_RING_START_FROM_SNAPSHOT, W)
                        for s in range(kv.sessions)], verify=True)
    torch.cuda.synchronize()
    j = torch.arange(W, device=dev)
    for s in range(kv.sessions):
        slot = (kv.ring_start[s] + j) % W
        a = kv.page_table[s].long()[:, slot // P]
        b = pt2[s].long()[:, slot // P]
        assert torch.equal(kv.k_pool[a, slot % P], k2[b, slot % P]), s
        assert torch.equal(kv.v_pool[a, slot % P], v2[b, slot % P]), s
    assert torch.equal(m2, kv.meta)
    for x in snaps:
        ctx.delete(x)


def test_prepared_host_calls_track_current_bytes(ctx, dev):
    n = 8
    obs, rng = _markov(n, dev, 910)
    arr = ctx.session_array([pcs.markov_session(s, obs[s], rng[s]) for s in range(n)])
    cplan, hs = ctx.plan_checkpoint(arr, n, pcs.PCS_PLACE_PINNED_HOST)
    o2, r2 = torch.zeros_like(obs), torch.zeros_like(rng)
    tarr = ctx.session_array([pcs.markov_session(s, o2[s], r2[s]) for s in range(n)])
    rplan = ctx.plan_restore(hs, n, tarr, verify=2)
    for round_ in range(3):
        g = torch.Generator(device=dev).manual_seed(920 + round_)
        obs.copy_(torch.randint(0, 256, obs.shape, generator=g, device=dev, dtype=torch.uint8))
        rng[:, 1] += 1
        ctx.plan_run(cplan)
        ctx.plan_run(rplan)
        torch.cuda.synchronize()
        ctx.sync()
        assert torch.equal(o2, obs) and torch.equal(r2, rng), round_
        for s in (0, n - 1):
            assert np.array_equal(ctx.record(pcs.Snapshot(ctx, hs[s])).numpy(),
                                  _oracle_markov(s, obs, rng)), (round_, s)
    ctx.plan_destroy(rplan)
    ctx.plan_destroy(cplan)
    ctx.delete_raw(hs, n)


def test_corrupt_host_record_is_reported(ctx, dev, tmp_path):
    n = 8
    obs, rng = _markov(n, dev, 930)
    snaps = ctx.checkpoint([pcs.markov_session(s, obs[s], rng[s]) for s in range(n)],
                           placement=pcs.PCS_PLACE_PINNED_HOST)
    # One record with a flipped payload byte, read back into host memory.
    bad = ctx.record(snaps[5]).numpy().copy()
    bad[ctx.section(snaps[5], 0).offset + 4321] ^= 0x10
    path = str(tmp_path / "bad.pcs")
    bad.tofile(path)
    back = ctx.read_file(path, pcs.PCS_PLACE_PINNED_HOST)
    group = snaps[:5] + [back] + snaps[6:]
    o2, r2 = torch.zeros_like(obs), torch.zeros_like(rng)
    st = ctx.restore_status(group, [pcs.markov_session(s, o2[s], r2[s]) for s in range(n)],
                            verify=True)
    assert st == pcs.PCS_E_CORRUPT
    for x in snaps + [back]:
        ctx.delete(x)
