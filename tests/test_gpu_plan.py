"""GPU parity: prepared checkpoint and restore (pcs_plan_*).

A prepared checkpoint rewrites its snapshots on every run, so after each run
the records equal the oracle's records of the sessions' current bytes; a
prepared restore writes the records' current bytes into its targets.  Plans
keep their records alive after the snapshot handles are deleted, order
themselves after readers on other streams, and refuse synchronous
verification.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth

pytestmark = pytest.mark.gpu


def _markov(n, dev, seed=600):
    ms = [synth.markov(seed=seed + i, shape=(3, 30 + i % 7, 41)) for i in range(n)]
    obs = [m.obs.to(dev) for m in ms]
    rng = [m.rng.to(dev) for m in ms]
    return obs, rng


def _oracle_rec(i, o, r):
    return oracle.pack(oracle.markov_session(i, o.cpu().numpy(),
                                             r.cpu().numpy().view(np.uint64)))


@pytest.mark.parametrize("n", [3, 70])  # the fused small-call kernel and the general path
def test_plan_checkpoint_tracks_current_bytes(ctx, dev, n):
    obs, rng = _markov(n, dev)
    arr = ctx.session_array([pcs.markov_session(i, obs[i], rng[i]) for i in range(n)])
    plan, hs = ctx.plan_checkpoint(arr, n)
    for round_ in range(3):
        ctx.sync()
        for i in range(n):
            assert np.array_equal(ctx.record(pcs.Snapshot(ctx, hs[i])).numpy(),
                                  _oracle_rec(i, obs[i], rng[i])), (round_, i)
        g = torch.Generator(device=dev).manual_seed(round_)
        for i in range(n):
            obs[i].copy_(torch.randint(0, 256, obs[i].shape, generator=g, device=dev,
                                       dtype=torch.uint8))
            rng[i][0] += 1
        ctx.plan_run(plan)
    ctx.delete_raw(hs, n)
    ctx.plan_destroy(plan)


def test_plan_restore_and_lifetime(ctx, dev):
    n = 40
    obs, rng = _markov(n, dev, seed=700)
    arr = ctx.session_array([pcs.markov_session(i, obs[i], rng[i]) for i in range(n)])
    cplan, hs = ctx.plan_checkpoint(arr, n)
    outs = [(torch.zeros_like(o), torch.zeros_like(r)) for o, r in zip(obs, rng)]
    tarr = ctx.session_array([pcs.markov_session(i, a, b) for i, (a, b) in enumerate(outs)])
    rplan = ctx.plan_restore(hs, n, tarr, verify=2)
    # The handles go; both plans keep the records.
    ctx.delete_raw(hs, n)
    for round_ in range(3):
        ctx.plan_run(rplan)
        ctx.sync()
        for (a, b), o, r in zip(outs, obs, rng):
            assert torch.equal(a, o) and torch.equal(b, r), round_
        for o in obs:
            o.add_(1)
        ctx.plan_run(cplan)
    ctx.plan_destroy(rplan)
    ctx.plan_destroy(cplan)
    with pytest.raises(pcs.PcsError) as e:
        ctx.plan_run(cplan)
    assert e.value.status == pcs.PCS_E_HANDLE


def test_plan_kv_matches_plain_calls(ctx, dev):
    kv = synth.kv(seed=91, sessions=3, layers=2, heads=16, head_dim=64, window=256,
                  page_rows=16, device=dev)
    src = ctx.session_array([pcs.kv_session(s, kv.meta[s], kv.k_pool, kv.v_pool, kv.page_table[s],
                                            kv.ring_start[s], kv.window) for s in range(3)])
    plan, hs = ctx.plan_checkpoint(src, 3)
    plain = ctx.checkpoint_raw(src, 3)
    ctx.sync()
    for i in range(3):
        assert np.array_equal(ctx.record(pcs.Snapshot(ctx, hs[i])).numpy(),
                              ctx.record(pcs.Snapshot(ctx, plain[i])).numpy())
    pt2 = synth.page_permutation(5, 3, 2, 16, device=dev)
    k2, v2, m2 = torch.zeros_like(kv.k_pool), torch.zeros_like(kv.v_pool), torch.zeros_like(kv.meta)
    dst = ctx.session_array([pcs.kv_session(s, m2[s], k2, v2, pt2[s],
                                            pcs.PCS_RING_START_FROM_SNAPSHOT, kv.window)
                             for s in range(3)])
    rplan = ctx.plan_restore(hs, 3, dst, verify=2)
    ctx.plan_run(rplan)
    ctx.sync()
    for s in range(3):
        for l in range(2):
            assert torch.equal(k2[pt2[s, l].long()], kv.k_pool[kv.page_table[s, l].long()])
            assert torch.equal(v2[pt2[s, l].long()], kv.v_pool[kv.page_table[s, l].long()])
    assert torch.equal(m2, kv.meta)
    ctx.plan_destroy(rplan)
    ctx.plan_destroy(plan)
    ctx.delete_raw(hs, 3)
    ctx.delete_raw(plain, 3)


def test_plan_checkpoint_waits_for_readers_on_other_streams(ctx, dev):
    n = 1 << 27
    x = torch.randint(0, 256, (n,), device=dev, dtype=torch.uint8)
    y = torch.zeros_like(x)
    sess = pcs.Session(1, pcs.PCS_KIND_MARKOV, [pcs.contig_section(pcs.PCS_SEC_OBS, x, dim0=n)],
                       keep=[x])
    arr = ctx.session_array([sess])
    plan, hs = ctx.plan_checkpoint(arr, 1)
    ctx.sync()
    want = x.clone()
    s2 = torch.cuda.Stream()
    tsess = pcs.Session(1, pcs.PCS_KIND_MARKOV, [pcs.contig_section(pcs.PCS_SEC_OBS, y, dim0=n)],
                        keep=[y])
    ctx.restore([pcs.Snapshot(ctx, hs[0])], [tsess], verify=2, stream=s2)
    x.add_(1)                      # on the current stream, after the first checkpoint
    ctx.plan_run(plan)             # must not overwrite the record before the restore read it
    torch.cuda.synchronize()
    ctx.sync()
    assert torch.equal(y, want)
    ctx.plan_destroy(plan)
    ctx.delete_raw(hs, 1)


def test_plan_argument_errors(ctx, dev):
    obs, rng = _markov(2, dev, seed=800)
    arr = ctx.session_array([pcs.markov_session(i, obs[i], rng[i]) for i in range(2)])
    plan, hs = ctx.plan_checkpoint(arr, 2)
    with pytest.raises(pcs.PcsError) as e:
        ctx.plan_restore(hs, 2, arr, verify=1)
    assert e.value.status == pcs.PCS_E_INVAL
    ctx.plan_destroy(plan)
    ctx.delete_raw(hs, 2)


@pytest.mark.parametrize("n", [3, 70])  # the fused small-call kernel and the general path
def test_calls_on_two_streams_run_side_by_side(ctx, dev, n):
    # Plain calls on two streams have a workspace each, and prepared calls a
    # buffer each, so nothing orders them against each other: many rounds on
    # both streams at once, nothing synchronised in between, every record
    # and every restored byte as the oracle says.
    streams = [torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)]
    sets = [_markov(n, dev, seed=800 + 100 * k) for k in range(2)]
    arrs = [ctx.session_array([pcs.markov_session(i, o[i], r[i]) for i in range(n)])
            for o, r in sets]
    outs = [[(torch.zeros_like(o), torch.zeros_like(r)) for o, r in zip(*sets[k])]
            for k in range(2)]
    tarrs = [ctx.session_array([pcs.markov_session(i, a, b) for i, (a, b) in enumerate(outs[k])])
             for k in range(2)]
    plans = []
    for k in range(2):
        cp, phs = ctx.plan_checkpoint(arrs[k], n, stream=streams[k])
        plans.append((cp, phs, ctx.plan_restore(phs, n, tarrs[k], verify=2)))
    torch.cuda.synchronize()
    kept = []
    for round_ in range(6):
        for k in range(2):
            hs = ctx.checkpoint_raw(arrs[k], n, stream=streams[k])
            ctx.restore_raw(hs, n, tarrs[k], verify=2, stream=streams[k])
            kept.append((k, hs))
            ctx.plan_run(plans[k][0], stream=streams[k])
            ctx.plan_run(plans[k][2], stream=streams[k])
    torch.cuda.synchronize()
    ctx.sync()  # no verified restore failed, no kernel error
    for k in range(2):
        obs, rng = sets[k]
        for i in range(n):
            assert torch.equal(outs[k][i][0], obs[i]) and torch.equal(outs[k][i][1], rng[i])
            want = _oracle_rec(i, obs[i], rng[i])
            assert np.array_equal(ctx.record(pcs.Snapshot(ctx, plans[k][1][i])).numpy(), want)
    for k, hs in kept[-2:]:
        for i in (0, n - 1):
            assert np.array_equal(ctx.record(pcs.Snapshot(ctx, hs[i])).numpy(),
                                  _oracle_rec(i, sets[k][0][i], sets[k][1][i]))
    for k, hs in kept:
        ctx.delete_raw(hs, n)
    for cp, phs, rp in plans:
        ctx.plan_destroy(rp)
        ctx.plan_destroy(cp)
        ctx.delete_raw(phs, n)
