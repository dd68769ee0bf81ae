"""Run one workload of the PCS hot path once (for profiling a single kernel).

    python profile_cases.py kv --sessions 8
    python profile_cases.py suspend --sessions 8
    python profile_cases.py classify --n 200 --hi-mib 32
    python profile_cases.py prune --sessions 256
    python profile_cases.py markov --sessions 4096
    python profile_cases.py markov_prepared --sessions 4096
    python profile_cases.py banks2 --sessions 64
    python profile_cases.py markov_layouts --sessions 4096
    python profile_cases.py mismatch --n 200 --hi-mib 32
    python profile_cases.py prune_global --sessions 256
    python profile_cases.py cow --sessions 64
    python profile_cases.py reads --n 200 --hi-mib 32
    python profile_cases.py topk --sessions 2048

Each case builds its seeded synthetic population on cuda:0, runs the step
`--warmup` times, then once more, and prints the device time of that last
run.  Intended to be run under a profiler with the launch count of the
warm-up runs skipped.
"""
from __future__ import annotations

import argparse
import json

import torch

from paper_2607_21686_gb300 import build, pcs, synth


def _timed(fn, warmup):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1)


def case_kv(ctx, a, dev):
    kv = synth.kv(sessions=a.sessions, device=dev)
    pt2 = synth.page_permutation(7, kv.sessions, kv.layers, kv.window // kv.page_rows, device=dev)
    k2, v2, m2 = torch.empty_like(kv.k_pool), torch.empty_like(kv.v_pool), torch.empty_like(kv.meta)
    src = ctx.session_array([pcs.kv_session(s, kv.meta[s], kv.k_pool, kv.v_pool, kv.page_table[s],
                                            kv.ring_start[s], kv.window) for s in range(kv.sessions)])
    dst = ctx.session_array([pcs.kv_session(s, m2[s], k2, v2, pt2[s],
                                            pcs.PCS_RING_START_FROM_SNAPSHOT, kv.window)
                             for s in range(kv.sessions)])

    def step():
        hs = ctx.checkpoint_raw(src, kv.sessions)
        ctx.restore_raw(hs, kv.sessions, dst, verify=2)
        ctx.delete_raw(hs, kv.sessions)
    return _timed(step, a.warmup)


def case_suspend(ctx, a, dev):
    """The KV sessions across the host link: checkpoint into records in
    pinned host memory, then a verified restore from them into a freshly
    permuted pool."""
    kv = synth.kv(sessions=a.sessions, device=dev)
    pt2 = synth.page_permutation(7, kv.sessions, kv.layers, kv.window // kv.page_rows, device=dev)
    k2, v2, m2 = torch.empty_like(kv.k_pool), torch.empty_like(kv.v_pool), torch.empty_like(kv.meta)
    src = ctx.session_array([pcs.kv_session(s, kv.meta[s], kv.k_pool, kv.v_pool, kv.page_table[s],
                                            kv.ring_start[s], kv.window) for s in range(kv.sessions)])
    dst = ctx.session_array([pcs.kv_session(s, m2[s], k2, v2, pt2[s],
                                            pcs.PCS_RING_START_FROM_SNAPSHOT, kv.window)
                             for s in range(kv.sessions)])

    def step():
        hs = ctx.checkpoint_raw(src, kv.sessions, pcs.PCS_PLACE_PINNED_HOST)
        ctx.restore_raw(hs, kv.sessions, dst, verify=2)
        ctx.delete_raw(hs, kv.sessions)
    return _timed(step, a.warmup)


def case_classify(ctx, a, dev):
    sw = synth.sweep(n=a.n, hi=a.hi_mib << 20, device=dev)
    fp0 = ctx.fingerprint(sw.before)
    arr = ctx.buf_array(sw.after)
    must = torch.empty(len(sw.after), dtype=torch.uint8, device=dev)
    fp1 = torch.empty(len(sw.after), dtype=torch.int64, device=dev)
    return _timed(lambda: ctx.classify(arr, fp0, fp1, must), a.warmup)


def case_prune(ctx, a, dev):
    b = synth.banks_config5(sessions=a.sessions, device=dev)
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]] for s in range(b.sessions)]
    banks = ctx.banks_array(keys, [b.queries[s] for s in range(b.sessions)], 1024 + 2048)
    params = ctx.params(pcs.PCS_K_BUDGET, budget=int(sum(b.n) * 3072 * 0.627))
    ks = ctx.prune_counts(banks, b.sessions, params)
    kept = torch.empty(sum(ks), dtype=torch.int32, device=dev)
    return _timed(lambda: ctx.prune(banks, b.sessions, params, kept), a.warmup)


def case_markov(ctx, a, dev):
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(1))
    obs = torch.randint(0, 256, (a.sessions, 3, 256, 256), generator=g, device=dev, dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (a.sessions, 2), generator=g, device=dev, dtype=torch.int64)
    arr = ctx.session_array([pcs.markov_session(s, obs[s], rng[s]) for s in range(a.sessions)])

    def step():
        hs = ctx.checkpoint_raw(arr, a.sessions)
        ctx.restore_raw(hs, a.sessions, arr)
        ctx.delete_raw(hs, a.sessions)
    return _timed(step, a.warmup)


def case_markov_prepared(ctx, a, dev):
    # The Markov batch as prepared calls: checkpoint, then verified restore
    # (mismatches counted on the device), launches only.
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(1))
    obs = torch.randint(0, 256, (a.sessions, 3, 256, 256), generator=g, device=dev, dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (a.sessions, 2), generator=g, device=dev, dtype=torch.int64)
    arr = ctx.session_array([pcs.markov_session(s, obs[s], rng[s]) for s in range(a.sessions)])
    cplan, hs = ctx.plan_checkpoint(arr, a.sessions)
    rplan = ctx.plan_restore(hs, a.sessions, arr, verify=2)

    def step():
        ctx.plan_run(cplan)
        ctx.plan_run(rplan)
    ms = _timed(step, a.warmup)
    ctx.sync()
    ctx.plan_destroy(rplan)
    ctx.plan_destroy(cplan)
    ctx.delete_raw(hs, a.sessions)
    return ms


def case_banks2(ctx, a, dev):
    # Memory banks (64 by default): prune to k = min(n, 128), checkpoint the
    # kept entries to HBM, verified restore into compacted banks, delete.
    b = synth.banks_config2(device=dev, sessions=a.sessions)
    S = b.sessions
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    vals = [b.values[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    banks = ctx.banks_array(keys, [b.queries[s] for s in range(S)], 512 + b.value_bytes)
    # Kept lists on 16-byte boundaries, as in bench.py's bank row.
    params = ctx.params(pcs.PCS_K_FIXED, k_max=128, kept_align=4)
    ks = ctx.prune_counts(banks, S, params)
    koff = [0]
    for k in ks:
        koff.append(koff[-1] + (k + 3) // 4 * 4)
    kept = torch.empty(koff[-1], dtype=torch.int32, device=dev)
    sarr = ctx.session_array([pcs.bank_session(s, keys[s], vals[s], kept[koff[s]:koff[s] + ks[s]])
                              for s in range(S)])
    outs = [(torch.empty(ks[s], dtype=torch.int32, device=dev),
             torch.empty(ks[s], 256, dtype=torch.float16, device=dev),
             torch.empty((ks[s],) + tuple(b.values.shape[1:]), dtype=b.values.dtype, device=dev))
            for s in range(S)]
    tarr = ctx.session_array([pcs.bank_targets(s, *outs[s]) for s in range(S)])

    def step():
        ctx.prune(banks, S, params, kept)
        hs = ctx.checkpoint_raw(sarr, S)
        ctx.restore_raw(hs, S, tarr, verify=2)
        ctx.delete_raw(hs, S)
    return _timed(step, a.warmup)


def case_markov_layouts(ctx, a, dev):
    # The same observation bytes packed twice: as one contiguous section per
    # session, then as the same tensor addressed through 32 KiB rows
    # (identity row index).  Records, sizes and addresses are identical; only
    # the kernel's staging path differs.
    rows_per = 196608 // 32768
    pool = torch.randint(0, 256, (a.sessions * rows_per, 32768), device=dev, dtype=torch.uint8)
    flat = pool.view(a.sessions, 196608)
    idx = torch.arange(a.sessions * rows_per, dtype=torch.int32, device=dev)
    contig = ctx.session_array([pcs.Session(s, pcs.PCS_KIND_MARKOV,
                                            [pcs.contig_section(pcs.PCS_SEC_OBS, flat[s])],
                                            keep=[pool]) for s in range(a.sessions)])
    rows = ctx.session_array([pcs.Session(s, pcs.PCS_KIND_MARKOV,
                                          [pcs.rows_section(pcs.PCS_SEC_OBS, pool,
                                                            idx[rows_per * s:rows_per * (s + 1)])],
                                          keep=[pool, idx]) for s in range(a.sessions)])

    def step():
        for arr in (contig, rows):
            ctx.delete_raw(ctx.checkpoint_raw(arr, a.sessions), a.sessions)
    return _timed(step, a.warmup)


def case_mismatch(ctx, a, dev):
    sw = synth.sweep(n=a.n, hi=a.hi_mib << 20, device=dev)
    b0, b1 = ctx.buf_array(sw.before), ctx.buf_array(sw.after)
    counts = torch.empty(len(sw.after), dtype=torch.int64, device=dev)
    return _timed(lambda: ctx.mismatch(b0, b1, counts), a.warmup)


def case_prune_global(ctx, a, dev):
    b = synth.banks_config5(sessions=a.sessions, device=dev)
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]] for s in range(b.sessions)]
    banks = ctx.banks_array(keys, [b.queries[s] for s in range(b.sessions)], 1024 + 2048)
    kept = torch.empty(sum(b.n), dtype=torch.int32, device=dev)
    koff = torch.empty(b.sessions + 1, dtype=torch.int32, device=dev)
    budget = int(sum(b.n) * 3072 * 0.627)
    return _timed(lambda: ctx.prune_global(banks, b.sessions, budget, kept, koff), a.warmup)


def case_cow(ctx, a, dev):
    # Every session's K and V pages shared by a fork, then the copy leg of one
    # page per layer and K/V of each child.
    S, layers, per = a.sessions, 24, 64
    live = S * 2 * layers * per
    pages = torch.empty(live + S * 2 * layers, 16, 16, 64, dtype=torch.bfloat16, device=dev)
    pool = pcs.Pool(ctx, pages)
    parent = pool.alloc(live)
    child = torch.empty_like(parent)
    ent = (torch.arange(S * 2 * layers) * per + 5).to(torch.int32).to(dev)

    def step():
        pool.share(parent, child)
        pool.prepare_write(child, ent)
        pool.release(child)
    ms = _timed(step, a.warmup)
    pool.destroy()
    return ms


def case_reads(ctx, a, dev):
    # A read log over the sweep's buffers: 140 of them read, 60 never.
    sw = synth.sweep(n=a.n, hi=a.hi_mib << 20, device=dev)
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(4) + 9)
    bases = torch.tensor([t.data_ptr() for t in sw.after], dtype=torch.int64, device=dev)
    lens = torch.tensor([t.numel() * t.element_size() for t in sw.after], dtype=torch.int64,
                        device=dev)
    m = 1 << 24
    which = torch.randint(0, int(0.7 * len(sw.after)), (m,), generator=g, device=dev)
    off = (torch.rand(m, generator=g, device=dev) * lens[which]).long()
    nbytes = torch.minimum(torch.randint(1, 4097, (m,), generator=g, device=dev,
                                         dtype=torch.int64), lens[which] - off)
    arr = ctx.buf_array(sw.after)
    flags = torch.empty(len(sw.after), dtype=torch.uint8, device=dev)
    addr = bases[which] + off
    return _timed(lambda: ctx.classify_reads(arr, addr, nbytes, flags), a.warmup)


def case_topk(ctx, a, dev):
    # Recency-keyed retention: last-use steps as rank keys, 62.7% kept per bank.
    b = synth.banks_config5(sessions=a.sessions, device=dev)
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(5) + 3)
    keys = torch.randint(0, 1 << 20, (sum(b.n),), generator=g, device=dev).float()
    k = [int(x * 0.627) for x in b.n]
    kept = torch.empty(sum(k), dtype=torch.int32, device=dev)
    na, ka = ctx.int32_array(b.n), ctx.int32_array(k)
    return _timed(lambda: ctx.topk(keys, na, ka, kept), a.warmup)


CASES = {"kv": case_kv, "suspend": case_suspend, "classify": case_classify, "prune": case_prune, "markov": case_markov,
         "markov_prepared": case_markov_prepared, "banks2": case_banks2,
         "markov_layouts": case_markov_layouts,
         "mismatch": case_mismatch, "prune_global": case_prune_global, "cow": case_cow,
         "reads": case_reads, "topk": case_topk}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("case", choices=sorted(CASES))
    ap.add_argument("--sessions", type=int, default=8)
    ap.add_argument("--n", type=int, default=200)
    ap.add_argument("--hi-mib", type=int, default=32)
    ap.add_argument("--warmup", type=int, default=1)
    a = ap.parse_args()
    build.build()
    dev = torch.device("cuda:0")
    torch.cuda.set_device(dev)
    with pcs.Context(0) as ctx:
        ms = CASES[a.case](ctx, a, dev)
        ctx.sync()
    print(json.dumps({"case": a.case, "ms": round(ms, 4)}))


if __name__ == "__main__":
    main()
