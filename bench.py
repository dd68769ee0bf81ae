"""Benchmark of the PCS hot path on GB300.

A step = one pass of the batched path over the windowed-KV population:
checkpoint of every session (gather of the paged ring into contiguous PCS1
records, fingerprint of every section fused into the copy, headers) and a
verified restore into a freshly permuted page pool (scatter, fingerprints
recomputed and checked), then delete.

Workload (default): 256 sessions x 24 layers x 16 heads x 64, bf16 K and V,
window 1024 tokens in 16-token pages randomly permuted in one pool, ring
start ~ U[0,1023].  Algorithmic bytes per step: pack reads and writes
25.77 GB, restore reads and writes 25.77 GB -> 103.1 GB.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl pcs|reference]
                    [--sessions S] [--layers L] [--no-cpu-baseline] [--no-e2e]

Prints one JSON line (rank 0).  Under torchrun each rank runs the same
workload on its own GPU (sessions are independent: weak scaling, no data
collective); the timing is the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "snapshot+restore GB/s and sessions/s on 1 GB300; % of HBM (PCIe) roofline"

# DRAM bytes (read + write) per launch of the streaming kernels, from the ncu
# capture summarised in profiles/k_bulk_kv8x24_full.md (8 sessions, scaled by
# sessions / 8), valid only for the streaming-kernel source it was taken on.
NCU_TRAFFIC = {
    "source_sha256_prefix": "82fadcb44e34aaa7",
    "sessions": 8,
    "k_bulk<pack>": 805706752 + 754244352,
    "k_bulk<restore_verify>": 805732608 + 754476544,
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="pcs", choices=["pcs", "reference"])
    ap.add_argument("--sessions", type=int, default=256)
    ap.add_argument("--layers", type=int, default=24)
    ap.add_argument("--heads", type=int, default=16)
    ap.add_argument("--head-dim", type=int, default=64)
    ap.add_argument("--window", type=int, default=1024)
    ap.add_argument("--page-rows", type=int, default=16)
    ap.add_argument("--no-verify", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-rows", action="store_true",
                    help="skip the per-row measurements on the other populations")
    return ap.parse_args()


def workload_name(a) -> str:
    return ("kv-window %d sessions x %d layers x %d heads x %d, bf16, window %d, %d-token pages"
            % (a.sessions, a.layers, a.heads, a.head_dim, a.window, a.page_rows))


def bench_config(a, world: int) -> dict:
    """The `config` of both arms' JSON lines (the same workload and settings)."""
    return {"workload": workload_name(a), "sessions": a.sessions * world, "layers": a.layers,
            "verify": not a.no_verify, "l2": "inputs larger than L2 (24 GiB pools)"}


def step_bytes(a) -> int:
    """Algorithmic bytes per step: pack R+W and restore R+W of every section."""
    sec = a.window * a.heads * a.head_dim * 2
    meta = 32
    payload = a.sessions * (2 * a.layers * sec + meta)
    return 4 * payload


def kernel_source_sha() -> str:
    """sha256 prefix of the streaming kernels' code: pcs_kernels.cu up to the
    finalisation kernels (helpers, the register kernel, the TMA kernel, the
    hash kernel), with // comments and blank lines left out, so that a change
    of wording does not disown a capture of the same code."""
    import hashlib
    import re
    p = os.path.join(ROOT, "paper_2607_21686_gb300", "csrc", "pcs_kernels.cu")
    with open(p, "rb") as f:
        text = f.read()
    cut = text.find(b"// Finalisation: stream fps")
    code = text[:cut if cut > 0 else len(text)].decode()
    lines = [re.sub(r"//.*$", "", ln).rstrip() for ln in code.splitlines()]
    code = "\n".join(ln for ln in lines if ln.strip())
    return hashlib.sha256(code.encode()).hexdigest()[:16]


def ncu_traffic(kernel: str, sessions: int):
    """Measured DRAM traffic per launch scaled to `sessions`, or None."""
    if kernel not in NCU_TRAFFIC or kernel_source_sha() != NCU_TRAFFIC["source_sha256_prefix"]:
        return None
    return round(NCU_TRAFFIC[kernel] * sessions / NCU_TRAFFIC["sessions"])


def max_over_ranks(x: float) -> float:
    """The largest of one float across the ranks of the default process group."""
    if not torch.distributed.is_initialized() or torch.distributed.get_world_size() == 1:
        return x
    dev = "cpu"
    if torch.distributed.get_backend() == "nccl":
        dev = torch.device("cuda", torch.cuda.current_device())
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def load_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "source": "fallback"}


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# CPU oracle leg (bounded sample of the same workload)
# ---------------------------------------------------------------------------

def _oracle_sessions(geom, seconds: float):
    """Whole sessions through the oracle (checkpoint + verified restore) for
    about `seconds` on this process's core: (sessions done, elapsed s)."""
    import numpy as np

    import oracle
    from paper_2607_21686_gb300 import synth

    a = argparse.Namespace(**geom)
    pages = a.window // a.page_rows
    kv = synth.kv(seed=synth.seed_for(3), sessions=1, layers=a.layers, heads=a.heads,
                  head_dim=a.head_dim, window=a.window, page_rows=a.page_rows, device="cpu")
    kp = kv.k_pool.view(torch.int16).numpy().view(np.uint16)
    vp = kv.v_pool.view(torch.int16).numpy().view(np.uint16)
    pt = kv.page_table[0].numpy()
    pt2 = synth.page_permutation(7, 1, a.layers, pages)[0].numpy()
    kp2, vp2 = np.zeros_like(kp), np.zeros_like(vp)
    meta = kv.meta[0].numpy().copy()
    meta2 = np.zeros_like(meta)
    done, t0 = 0, time.perf_counter()
    while True:
        rec = oracle.pack(oracle.kv_session(0, meta, kp, vp, pt, kv.ring_start[0], a.window,
                                            a.page_rows, kv.row_bytes))
        t = oracle.kv_session(0, meta2, kp2, vp2, pt2, 0, a.window, a.page_rows, kv.row_bytes,
                              ring_start_override=oracle.RING_START_FROM_RECORD)
        assert oracle.restore(rec, t, verify=True) == 0
        done += 1
        el = time.perf_counter() - t0
        if el >= seconds or done >= 64:
            break
    return done, el


def oracle_pool(procs: int):
    """Worker processes for the oracle (spawn: this process may hold a CUDA
    context), or None for one core."""
    import multiprocessing as mp

    import oracle

    oracle.build()  # once, before any worker loads it
    return mp.get_context("spawn").Pool(procs) if procs > 1 else None


def cpu_oracle_rate(a, seconds: float, pool=None) -> dict:
    """Oracle checkpoint + verified restore of whole, independent sessions,
    about `seconds` on each core: one core, or one per worker of `pool`."""
    import oracle

    oracle.build()
    geom = {k: getattr(a, k) for k in ("layers", "heads", "head_dim", "window", "page_rows",
                                       "sessions")}
    per_session = step_bytes(a) // a.sessions
    procs = pool._processes if pool is not None else 1
    if pool is None:
        done, el = _oracle_sessions(geom, seconds)
    else:
        res = pool.starmap(_oracle_sessions, [(geom, seconds)] * procs)
        done, el = sum(r[0] for r in res), max(r[1] for r in res)
    gbs = done * per_session / el / 1e9
    return {"value": round(gbs, 4), "unit": "GB/s", "cores": procs, "kind": "oracle",
            "sample": "%d whole session(s) of the same geometry (checkpoint + verified restore, "
                      "%.1f MB each) on %d core(s), %.1f s" % (done, per_session / 1e6, procs, el),
            "sessions_per_s": round(done / el, 4)}


def host_cores() -> int:
    return len(os.sched_getaffinity(0))


# ---------------------------------------------------------------------------
# GPU leg
# ---------------------------------------------------------------------------

def run_reference(a, rank, world):
    """The oracle timed on the host cores: K steps of a bounded sample each."""
    if rank != 0:
        return None
    per_step = max(1.0, min(a.cpu_seconds, 120.0 / max(1, a.steps + a.warmup)))
    pool = oracle_pool(host_cores())
    try:
        for _ in range(a.warmup):
            cpu_oracle_rate(a, per_step / 4, pool)
        rates = [cpu_oracle_rate(a, per_step, pool) for _ in range(a.steps)]
    finally:
        if pool is not None:
            pool.close()
            pool.join()
    v = statistics.median(r["value"] for r in rates)
    sps = statistics.median(r["sessions_per_s"] for r in rates)
    line = {"metric": METRIC, "value": v, "unit": "GB/s", "n_gpus": world, "steps": a.steps,
            "warmup": a.warmup, "ms_per_step": round(a.sessions / sps * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u64",
            "data": "synthetic", "impl": "reference",
            "config": bench_config(a, world),
            "sessions_per_s": sps,
            "cpu_baseline": dict(rates[-1], value=v),
            "e2e": {"value": v, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    return line


def bind_host_to_gpu(device: int) -> str:
    """Run on the host CPUs next to the GPU, so that pinned buffers (first
    touched here) sit on the GPU's NUMA node; the host link is slower from
    the other node.  Returns the CPU list bound to, or why not."""
    try:
        p = torch.cuda.get_device_properties(device)
        base = "/sys/bus/pci/devices/%04x:%02x:%02x.0" % (p.pci_domain_id, p.pci_bus_id,
                                                         p.pci_device_id)
        with open(base + "/local_cpulist") as f:
            spec = f.read().strip()
        cpus = set()
        for part in spec.split(","):
            lo, _, hi = part.partition("-")
            cpus.update(range(int(lo), int(hi or lo) + 1))
        cpus &= os.sched_getaffinity(0)
        if not cpus:
            return "unbound: no local CPU available to this process"
        os.sched_setaffinity(0, cpus)
        return spec
    except (OSError, ValueError, AttributeError) as ex:
        return "unbound: %s" % ex


def run_pcs(a, rank, world, local_rank):
    from paper_2607_21686_gb300 import build, pcs, synth

    build.build()
    host_cpus = bind_host_to_gpu(local_rank)
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    ctx = pcs.Context(local_rank)
    stream = torch.cuda.current_stream()
    pages = a.window // a.page_rows

    kv = synth.kv(seed=synth.seed_for(3) + 1000 * rank, sessions=a.sessions, layers=a.layers,
                  heads=a.heads, head_dim=a.head_dim, window=a.window, page_rows=a.page_rows,
                  device=dev)
    pt2 = synth.page_permutation(synth.seed_for(3) + 7, a.sessions, a.layers, pages, device=dev)
    k2, v2 = torch.empty_like(kv.k_pool), torch.empty_like(kv.v_pool)
    meta2 = torch.empty_like(kv.meta)
    src = [pcs.kv_session(s, kv.meta[s], kv.k_pool, kv.v_pool, kv.page_table[s], kv.ring_start[s],
                          a.window) for s in range(a.sessions)]
    dst = [pcs.kv_session(s, meta2[s], k2, v2, pt2[s], pcs.PCS_RING_START_FROM_SNAPSHOT,
                          a.window) for s in range(a.sessions)]
    src_arr, dst_arr = ctx.session_array(src), ctx.session_array(dst)
    # Verification runs on the device inside the restore kernels; mismatches
    # are reported by the pcs_sync after the timed region (verify mode 2).
    verify = 0 if a.no_verify else 2
    S = a.sessions

    def step():
        hs = ctx.checkpoint_raw(src_arr, S)
        ctx.restore_raw(hs, S, dst_arr, verify=verify)
        ctx.delete_raw(hs, S)

    for _ in range(a.warmup):
        step()
    ctx.sync()
    # Spot-check the restore of the warm-up (full parity lives in the tests).
    s0 = 0
    j = torch.arange(a.window, device=dev)
    slot = (kv.ring_start[s0] + j) % a.window
    for l in (0, a.layers - 1):
        orig = kv.k_pool[kv.page_table[s0, l].long()[slot // a.page_rows], slot % a.page_rows]
        back = k2[pt2[s0, l].long()[slot // a.page_rows], slot % a.page_rows]
        assert torch.equal(orig, back), "restore mismatch"

    launches0 = ctx.stats().kernel_launches
    ctx.timing(True)
    clocks = ClockSampler(local_rank)
    clocks.start()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(a.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop()
    ctx.sync()  # raises if any verified restore of the timed steps failed
    ms = e0.elapsed_time(e1)
    ktimes = ctx.kernel_times()
    ctx.timing(False)
    launches = ctx.stats().kernel_launches - launches0
    ms = max_over_ranks(ms)

    # End to end through the public API with the state coming from host memory.
    e2e = None
    if not a.no_e2e:
        if world > 1:
            torch.distributed.barrier()
        e2e = run_e2e(a, ctx, kv, dst, stream, dev)
        if world > 1:
            e2e = e2e_over_ranks(a, e2e, world)

    rows = None
    if not a.no_rows and rank == 0:
        rows = {"fork": measure_fork(ctx, src, stream),
                "kv_suspend_resume": measure_suspend_resume(a, ctx, src, dst, stream, dev,
                                                            steps=5)}
        del src, dst, kv, k2, v2, meta2
        torch.cuda.empty_cache()
        rows.update(run_rows(ctx, dev, stream))

    res = {"ms": ms, "ktimes": ktimes, "launches": launches, "clocks": clk, "e2e": e2e,
           "rows": rows, "host_cpus": host_cpus}
    ctx.close()
    return res


# ---------------------------------------------------------------------------
# The other rows of the path, each on its own population (informational;
# the headline `value` above is the KV checkpoint + restore step)
# ---------------------------------------------------------------------------

def _loop_ms(fn, stream, calls=10, warm=2):
    """Device time per call of `calls` back-to-back calls between one pair of
    events: the throughput of a repeated step (the host prepares call i+1
    while the GPU runs call i), timed as the headline step is."""
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(calls):
        fn()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / calls


def _events_ms(fn, stream, reps=5, warm=2):
    """Best and median device time of fn() over reps, CUDA events on `stream`."""
    for _ in range(warm):
        fn()
    torch.cuda.synchronize()
    ts = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    ts.sort()
    return ts[0], ts[len(ts) // 2]


def measure_link(dev, stream) -> dict:
    """The host link with pinned cudaMemcpyAsync of 1 GiB (best of 5): each
    direction alone, and both at once on two streams (per direction)."""
    x = torch.empty(1 << 30, dtype=torch.uint8, pin_memory=True)
    x2 = torch.empty(1 << 30, dtype=torch.uint8, pin_memory=True)
    y = torch.empty(1 << 30, dtype=torch.uint8, device=dev)
    y2 = torch.empty(1 << 30, dtype=torch.uint8, device=dev)
    h2d = (1 << 30) / (_events_ms(lambda: y.copy_(x, non_blocking=True), stream)[0] / 1e3) / 1e9
    d2h = (1 << 30) / (_events_ms(lambda: x.copy_(y, non_blocking=True), stream)[0] / 1e3) / 1e9
    other = torch.cuda.Stream(device=dev)

    def both():
        other.wait_stream(stream)
        y.copy_(x, non_blocking=True)
        with torch.cuda.stream(other):
            x2.copy_(y2, non_blocking=True)
        stream.wait_stream(other)
    duplex = (1 << 30) / (_events_ms(both, stream)[0] / 1e3) / 1e9
    del x, x2, y, y2
    return {"h2d_GBs": round(h2d, 1), "d2h_GBs": round(d2h, 1),
            "duplex_GBs_each_way": round(duplex, 1),
            "how": "pinned cudaMemcpyAsync 1 GiB, best of 5; duplex: one copy each way at once"}


def measure_fork(ctx, src, stream):
    """a9: fork every snapshot of the KV step in one call (independent copies)."""
    arr = ctx.session_array(src)
    n = len(src)
    hs = ctx.checkpoint_raw(arr, n)
    nbytes = sum(ctx.info(pcs_snapshot(ctx, hs[i])).total_bytes for i in range(n))

    def fork_all():
        ctx.delete_raw(ctx.fork_raw(hs, n), n)
    med = _loop_ms(fork_all, stream, calls=5, warm=1)
    ctx.delete_raw(hs, n)
    peak = load_peaks()["hbm_gbs"]
    gbs = 2 * nbytes / (med / 1e3) / 1e9
    return {"population": "256 KV snapshots (96 MiB each), one pcs_fork_many call",
            "bytes_rw": 2 * nbytes, "ms": round(med, 3), "GBs": round(gbs, 1),
            "frac_of_hbm": round(gbs / peak, 4)}


def pcs_snapshot(ctx, handle):
    from paper_2607_21686_gb300 import pcs
    return pcs.Snapshot(ctx, handle)


def run_rows(ctx, dev, stream):
    from paper_2607_21686_gb300 import pcs, synth

    peak = load_peaks()["hbm_gbs"]
    out = {}
    out["host_link"] = measure_link(dev, stream)
    h2d, d2h = out["host_link"]["h2d_GBs"], out["host_link"]["d2h_GBs"]

    # a1-a3: classification sweep, 200 buffers of 64 B .. 256 MiB.
    sw = synth.sweep(device=dev)
    tot = sum(sw.sizes)
    fp0 = ctx.fingerprint(sw.before)
    # Prebuilt buffer arrays and outputs: the timed region holds the call's
    # own work, not the binding's per-tensor marshalling.
    after_arr, before_arr = ctx.buf_array(sw.after), ctx.buf_array(sw.before)
    must = torch.empty(len(sw.after), dtype=torch.uint8, device=dev)
    fp1 = torch.empty(len(sw.after), dtype=torch.int64, device=dev)
    med = _loop_ms(lambda: ctx.classify(after_arr, fp0, fp1, must), stream)
    ctx.classify(after_arr, fp0, fp1, must)
    flips_ok = must.cpu().tolist() == [1 if f else 0 for f in sw.flipped]
    gbs = tot / (med / 1e3) / 1e9
    out["classify"] = {"population": "200 buffers, log-uniform 64 B..256 MiB, 60 flipped",
                       "bytes_read": tot, "ms": round(med, 3), "GBs": round(gbs, 1),
                       "frac_of_hbm": round(gbs / peak, 4), "flags_match_ground_truth": flips_ok}
    # The discovery distance on the same pairs: differing bytes of before / after.
    counts = torch.empty(len(sw.after), dtype=torch.int64, device=dev)
    med = _loop_ms(lambda: ctx.mismatch(before_arr, after_arr, counts), stream)
    mm_ok = ctx.mismatch(before_arr, after_arr, counts).cpu().tolist() == \
        [1 if f else 0 for f in sw.flipped]
    gbs = 2 * tot / (med / 1e3) / 1e9
    out["mismatch"] = {"population": "the same 200 buffer pairs (before, after)",
                       "bytes_read": 2 * tot, "ms": round(med, 3), "GBs": round(gbs, 1),
                       "frac_of_hbm": round(gbs / peak, 4), "counts_match_ground_truth": mm_ok}
    # State versus witness: a read log of 16M byte ranges (what a resume
    # touched) against the same 200 buffers.
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(4) + 9)
    bases = torch.tensor([t.data_ptr() for t in sw.after], dtype=torch.int64, device=dev)
    lens = torch.tensor([t.numel() * t.element_size() for t in sw.after], dtype=torch.int64,
                        device=dev)
    m = 1 << 24
    which = torch.randint(0, 140, (m,), generator=g, device=dev)  # 60 buffers never read
    off = (torch.rand(m, generator=g, device=dev) * lens[which]).long()
    addr = bases[which] + off
    nbytes = torch.minimum(torch.randint(1, 4097, (m,), generator=g, device=dev,
                                         dtype=torch.int64), lens[which] - off)  # within the buffer
    flags = torch.empty(len(sw.after), dtype=torch.uint8, device=dev)
    med = _loop_ms(lambda: ctx.classify_reads(after_arr, addr, nbytes, flags), stream)
    read_ok = flags.cpu().tolist()[140:] == [0] * 60 and all(flags.cpu().tolist()[:140])
    out["classify_reads"] = {"population": "16M reads (1 B-4 KiB) over 140 of the 200 buffers",
                             "reads": m, "ms": round(med, 3),
                             "Mreads_per_s": round(m / (med / 1e3) / 1e6, 1),
                             "GBs_of_log": round(16 * m / (med / 1e3) / 1e9, 1),
                             "flags_match_ground_truth": read_ok}
    del sw, fp0, must, fp1, counts, after_arr, before_arr, addr, nbytes, which, bases, lens, off

    out["banks_config2"] = measure_banks_config2(ctx, dev, stream, peak)

    # a4-a5, a7, a10: 2048 banks, relevance top-k under an 8 GiB host budget,
    # pack to pinned host, verified restore to HBM.
    b = synth.banks_config5(device=dev)
    S = b.sessions
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    vals = [b.values[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    qs = [b.queries[s] for s in range(S)]
    banks = ctx.banks_array(keys, qs, 1024 + 2048)
    params = ctx.params(pcs.PCS_K_BUDGET, budget=8 << 30)
    ks = ctx.prune_counts(banks, S, params)
    kept = torch.empty(sum(ks), dtype=torch.int32, device=dev)
    koff = torch.empty(S + 1, dtype=torch.int32, device=dev)
    kb = b.keys.numel() * b.keys.element_size()
    med = _loop_ms(lambda: ctx.prune(banks, S, params, kept, koff), stream)
    gbs = kb / (med / 1e3) / 1e9
    out["prune"] = {"population": "2048 banks, n ~ U[256,4096], key bf16[512]",
                    "key_bytes_read": kb, "ms": round(med, 3), "GBs": round(gbs, 1),
                    "frac_of_hbm": round(gbs / peak, 4), "kept_fraction": round(sum(ks) / sum(b.n), 4)}
    # The same banks under one relevance threshold across all of them.
    gkept = torch.empty(sum(b.n), dtype=torch.int32, device=dev)
    gkoff = torch.empty(S + 1, dtype=torch.int32, device=dev)
    medg = _loop_ms(lambda: ctx.prune_global(banks, S, 8 << 30, gkept, gkoff), stream)
    gk = int(gkoff[-1].item())
    out["prune_global"] = {
        "population": "the same 2048 banks, one threshold across all under 8 GiB",
        "key_bytes_read": kb, "ms": round(medg, 3), "GBs": round(kb / (medg / 1e3) / 1e9, 1),
        "frac_of_hbm": round(kb / (medg / 1e3) / 1e9 / peak, 4),
        "kept_fraction": round(gk / sum(b.n), 4),
        "kept_bytes": gk * (1024 + 2048)}
    del gkept, gkoff
    # Recency-keyed retention (lru): the same banks kept by last-use step.
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(5) + 3)
    last_use = torch.randint(0, 1 << 20, (sum(b.n),), generator=g, device=dev).float()
    rk = [int(x * 0.627) for x in b.n]
    rkept = torch.empty(sum(rk), dtype=torch.int32, device=dev)
    n_arr, k_arr = ctx.int32_array(b.n), ctx.int32_array(rk)
    med = _loop_ms(lambda: ctx.topk(last_use, n_arr, k_arr, rkept), stream)
    out["topk_recency"] = {"population": "the same 2048 banks, lru keys, 62.7% kept per bank",
                           "entries": sum(b.n), "ms": round(med, 3),
                           "Mentries_per_s": round(sum(b.n) / (med / 1e3) / 1e6, 1)}
    del last_use, rkept
    koff_h = koff.cpu().tolist()
    sess = [pcs.bank_session(s, keys[s], vals[s], kept[koff_h[s]:koff_h[s + 1]]) for s in range(S)]
    kept_bytes = sum(ks) * (1024 + 2048)
    outs = [(torch.empty(ks[s], dtype=torch.int32, device=dev),
             torch.empty(ks[s], 512, dtype=torch.bfloat16, device=dev),
             torch.empty(ks[s], 2048, dtype=torch.uint8, device=dev)) for s in range(S)]
    tg = [pcs.bank_targets(s, *outs[s]) for s in range(S)]
    # Prebuilt session arrays and handle arrays (the batch forms of the API),
    # verification on the device reported at the next sync.
    sarr, tarr = ctx.session_array(sess), ctx.session_array(tg)

    def ckpt_del():
        ctx.delete_raw(ctx.checkpoint_raw(sarr, S, pcs.PCS_PLACE_PINNED_HOST), S)
    med = _loop_ms(ckpt_del, stream, calls=3, warm=1)
    hs = ctx.checkpoint_raw(sarr, S, pcs.PCS_PLACE_PINNED_HOST)
    medr = _loop_ms(lambda: ctx.restore_raw(hs, S, tarr, verify=2), stream, calls=3, warm=1)
    ctx.sync()
    ctx.delete_raw(hs, S)
    out["suspend_to_host"] = {
        "population": "the 2048 pruned banks, %.2f GB kept" % (kept_bytes / 1e9),
        "ms": round(med, 3), "GBs": round(kept_bytes / (med / 1e3) / 1e9, 1),
        "frac_of_d2h_link": round(kept_bytes / (med / 1e3) / 1e9 / d2h, 4)}
    out["resume_from_host"] = {
        "population": "the same records, verified restore into HBM",
        "ms": round(medr, 3), "GBs": round(kept_bytes / (medr / 1e3) / 1e9, 1),
        "frac_of_h2d_link": round(kept_bytes / (medr / 1e3) / 1e9 / h2d, 4)}
    del b, keys, vals, outs, tg, sess, kept, sarr, tarr

    # Markovian sessions: one-session latency and a 4096-session batch.
    mk = synth.markov(device=dev)
    one = [pcs.markov_session(0, mk.obs, mk.rng)]
    oarr = ctx.session_array(one)
    for _ in range(20):
        ctx.delete_raw(ctx.checkpoint_raw(oarr, 1), 1)
    torch.cuda.synchronize()
    n = 1000
    t0 = time.perf_counter()
    for _ in range(n):
        ctx.delete_raw(ctx.checkpoint_raw(oarr, 1), 1)
    torch.cuda.synchronize()
    ck_us = (time.perf_counter() - t0) / n * 1e6
    h0 = ctx.checkpoint_raw(oarr, 1)
    t0 = time.perf_counter()
    for _ in range(n):
        ctx.restore_raw(h0, 1, oarr)
    torch.cuda.synchronize()
    rs_us = (time.perf_counter() - t0) / n * 1e6
    ctx.delete_raw(h0, 1)
    # One session as prepared calls: launches only.
    p1, ph = ctx.plan_checkpoint(oarr, 1)
    pr1 = ctx.plan_restore(ph, 1, oarr, verify=0)
    for _ in range(20):
        ctx.plan_run(p1)
        ctx.plan_run(pr1)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(n):
        ctx.plan_run(p1)
    torch.cuda.synchronize()
    pck_us = (time.perf_counter() - t0) / n * 1e6
    t0 = time.perf_counter()
    for _ in range(n):
        ctx.plan_run(pr1)
    torch.cuda.synchronize()
    prs_us = (time.perf_counter() - t0) / n * 1e6
    ctx.plan_destroy(pr1)
    ctx.plan_destroy(p1)
    ctx.delete_raw(ph, 1)
    g = torch.Generator(device=dev).manual_seed(synth.seed_for(1))
    obs = torch.randint(0, 256, (4096, 3, 256, 256), generator=g, device=dev, dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (4096, 2), generator=g, device=dev, dtype=torch.int64)
    batch = [pcs.markov_session(s, obs[s], rng[s]) for s in range(4096)]
    barr = ctx.session_array(batch)

    def batch_step():
        hs = ctx.checkpoint_raw(barr, 4096)
        ctx.restore_raw(hs, 4096, barr)
        ctx.delete_raw(hs, 4096)
    med = _loop_ms(batch_step, stream, calls=5, warm=1)
    # The same step as prepared calls: planned once, then launches only.
    cplan, phs = ctx.plan_checkpoint(barr, 4096)
    rplan = ctx.plan_restore(phs, 4096, barr, verify=2)

    def prepared_step():
        ctx.plan_run(cplan)
        ctx.plan_run(rplan)
    medp = _loop_ms(prepared_step, stream, calls=20, warm=2)
    ctx.sync()
    ctx.plan_destroy(rplan)
    ctx.plan_destroy(cplan)
    ctx.delete_raw(phs, 4096)
    out["markov"] = {"one_session_checkpoint_us": round(ck_us, 2),
                     "one_session_restore_us": round(rs_us, 2),
                     "one_session_prepared_checkpoint_us": round(pck_us, 2),
                     "one_session_prepared_restore_us": round(prs_us, 2),
                     "how": "wall clock per call (checkpoint incl. delete) through the ctypes "
                            "binding with a prebuilt session array, 1000 calls",
                     "paper_context_us": 12.0,
                     "batch_4096_sessions_per_s": round(4096 / (med / 1e3), 1),
                     "batch_GBs": round(4 * 4096 * (196608 + 16) / (med / 1e3) / 1e9, 1),
                     "prepared_4096_sessions_per_s": round(4096 / (medp / 1e3), 1),
                     "prepared_GBs": round(4 * 4096 * (196608 + 16) / (medp / 1e3) / 1e9, 1),
                     "prepared_frac_of_hbm": round(4 * 4096 * (196608 + 16) / (medp / 1e3) / 1e9
                                                   / peak, 4)}
    del obs, rng, batch, barr
    out["cow_fork"] = measure_cow_fork(ctx, dev, stream, peak)
    return out


def measure_banks_config2(ctx, dev, stream, peak):
    """a4-a5, a7-a10 on 64 memory banks: prune to k = min(n, 128) by relevance,
    checkpoint the kept entries to HBM, verified restore into compacted banks,
    delete -- one step, enqueued without a host wait (the kept counts are
    known on the host, so the sessions are described before the prune has
    written the indices they gather by)."""
    from paper_2607_21686_gb300 import pcs, synth

    b = synth.banks_config2(device=dev)
    S = b.sessions
    keys = [b.keys[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    vals = [b.values[b.entry_off[s]:b.entry_off[s + 1]] for s in range(S)]
    banks = ctx.banks_array(keys, [b.queries[s] for s in range(S)], 512 + b.value_bytes)
    # Each bank's kept list starts on a 16-byte boundary (kept_align 4), so the
    # checkpoint moves the lists with the other sections' bulk copies.
    params = ctx.params(pcs.PCS_K_FIXED, k_max=128, kept_align=4)
    ks = ctx.prune_counts(banks, S, params)
    koff = [0]
    for k in ks:
        koff.append(koff[-1] + (k + 3) // 4 * 4)
    kept = torch.empty(koff[-1], dtype=torch.int32, device=dev)
    sess = [pcs.bank_session(s, keys[s], vals[s], kept[koff[s]:koff[s] + ks[s]]) for s in range(S)]
    outs = [(torch.empty(ks[s], dtype=torch.int32, device=dev),
             torch.empty(ks[s], 256, dtype=torch.float16, device=dev),
             torch.empty((ks[s],) + tuple(b.values.shape[1:]), dtype=b.values.dtype, device=dev))
            for s in range(S)]
    sarr = ctx.session_array(sess)
    tarr = ctx.session_array([pcs.bank_targets(s, *outs[s]) for s in range(S)])

    def step():
        ctx.prune(banks, S, params, kept)
        hs = ctx.checkpoint_raw(sarr, S)
        ctx.restore_raw(hs, S, tarr, verify=2)
        ctx.delete_raw(hs, S)
    med = _loop_ms(step, stream, calls=20, warm=3)
    ctx.sync()
    # The restored banks hold exactly the kept rows, in ascending index.
    kept_h = kept.cpu()
    ok = True
    for s in (0, S // 2, S - 1):
        ki = kept_h[koff[s]:koff[s] + ks[s]]
        ok &= bool(torch.equal(outs[s][0].cpu(), ki)) and bool(torch.all(ki[1:] > ki[:-1]))
        ok &= bool(torch.equal(outs[s][2], vals[s][ki.long().to(dev)]))
    # Planned once, then launches only (prune, checkpoint, restore).
    cplan, phs = ctx.plan_checkpoint(sarr, S)
    rplan = ctx.plan_restore(phs, S, tarr, verify=2)

    def prepared_step():
        ctx.prune(banks, S, params, kept)
        ctx.plan_run(cplan)
        ctx.plan_run(rplan)
    medp = _loop_ms(prepared_step, stream, calls=20, warm=3)
    ctx.sync()
    ctx.plan_destroy(rplan)
    ctx.plan_destroy(cplan)
    ctx.delete_raw(phs, S)
    kb = sum(b.n) * 512
    payload = sum(ks) * (4 + 512 + b.value_bytes)
    moved = kb + 4 * payload
    return {"population": "64 banks, n ~ U[1,512], key fp16[256], latent bf16[16,32,32], "
                          "k = min(n,128); kept lists 16-byte aligned",
            "entries": sum(b.n), "kept": sum(ks), "key_bytes_read": kb,
            "bytes_per_step": moved, "how": "prune + checkpoint to HBM + verified restore + "
            "delete, 20 back-to-back steps between one pair of events",
            "ms": round(med, 4), "GBs": round(moved / (med / 1e3) / 1e9, 1),
            "sessions_per_s": round(S / (med / 1e3), 1),
            "frac_of_hbm": round(moved / (med / 1e3) / 1e9 / peak, 4),
            "prepared_ms": round(medp, 4),
            "prepared_GBs": round(moved / (medp / 1e3) / 1e9, 1),
            "prepared_sessions_per_s": round(S / (medp / 1e3), 1),
            "prepared_frac_of_hbm": round(moved / (medp / 1e3) / 1e9 / peak, 4),
            "restored_rows_match": ok}


def measure_cow_fork(ctx, dev, stream, peak):
    """Copy-on-write fork of the 256 KV sessions: share every K and V page
    (no bytes move), then the copy leg of each child's first token append
    (one page per layer and K/V: 12,288 page copies of 32 KiB)."""
    from paper_2607_21686_gb300 import pcs

    S, layers, per, page_rows = 256, 24, 64, 16
    live = S * 2 * layers * per
    spare = S * 2 * layers
    pages = torch.empty(live + spare, page_rows, 16, 64, dtype=torch.bfloat16, device=dev)
    pool = pcs.Pool(ctx, pages)
    parent = pool.alloc(live).view(S, 2, layers, per)
    g = torch.Generator().manual_seed(7)
    ring = torch.randint(0, per * page_rows, (S,), generator=g)
    # The ring page each child writes first, for every layer of K and V.
    ent = (torch.arange(S)[:, None] * (2 * layers * per) + torch.arange(2 * layers)[None, :] * per
           + (ring // page_rows)[:, None]).reshape(-1).to(torch.int32).to(dev)
    child = torch.empty_like(parent)
    page_bytes = pool.page_bytes

    fork_ms, write_ms = [], []
    for rep in range(7):
        e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        e[0].record(stream)
        pool.share(parent, child)
        e[1].record(stream)
        pool.prepare_write(child, ent)
        e[2].record(stream)
        pool.release(child)
        torch.cuda.synchronize()
        if rep >= 2:
            fork_ms.append(e[0].elapsed_time(e[1]))
            write_ms.append(e[1].elapsed_time(e[2]))
    ctx.sync()
    free = pool.query()[0]
    pool.destroy()
    del pages
    fork_ms.sort()
    write_ms.sort()
    fm, wm = fork_ms[len(fork_ms) // 2], write_ms[len(write_ms) // 2]
    moved = 2 * ent.numel() * page_bytes
    return {"population": "256 KV sessions (24 layers, K and V, 64 pages of 32 KiB each) "
                          "in one page pool",
            "fork_pages_shared": live, "fork_ms": round(fm, 4),
            "first_write_pages_copied": int(ent.numel()), "first_write_ms": round(wm, 4),
            "first_write_GBs": round(moved / (wm / 1e3) / 1e9, 1),
            "first_write_frac_of_hbm": round(moved / (wm / 1e3) / 1e9 / peak, 4),
            "pool_free_after": free, "pool_spare": spare}


def _anon_huge_bytes() -> int:
    """Anonymous memory the host kernel backs with huge pages (bytes)."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("AnonHugePages:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


class HostBuffer:
    """Pinned host memory on transparent huge pages: an anonymous mapping
    advised MADV_HUGEPAGE, touched, then page-locked with cudaHostRegister.
    With 64 KiB base pages, DMA over many GiB of small pages thrashes the
    host's address translation (one 12 GiB copy alternating with another ran
    at 159 GB/s instead of 211); huge pages keep the link at full rate."""

    def __init__(self, nbytes: int):
        import mmap
        self.n = nbytes
        self.mm = mmap.mmap(-1, nbytes, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
        if hasattr(mmap, "MADV_HUGEPAGE"):
            self.mm.madvise(mmap.MADV_HUGEPAGE)
        self.flat = torch.frombuffer(self.mm, dtype=torch.uint8)
        self.flat.fill_(0)
        self.addr = self.flat.data_ptr()
        rc = int(torch.cuda.cudart().cudaHostRegister(self.addr, nbytes, 0))
        if rc != 0:
            self.close()
            raise RuntimeError("cudaHostRegister failed (%d)" % rc)
        self.registered = True

    def view(self, shape, dtype):
        return self.flat.view(dtype).view(shape)

    def close(self):
        if getattr(self, "registered", False):
            torch.cuda.cudart().cudaHostUnregister(self.addr)
            self.registered = False
        self.flat = None
        if self.mm is not None:
            try:
                self.mm.close()
            except BufferError:  # views still alive; the mapping goes with them
                pass
            self.mm = None


def e2e_over_ranks(a, e2e: dict, world: int) -> dict:
    """The whole job's end-to-end line: every rank's step bytes over the
    slowest rank's time per step (all ranks ran their steps at once)."""
    ms = e2e.get("ms_per_step")
    if max_over_ranks(0.0 if ms is not None else 1.0) != 0.0:
        return {"value": None, "unit": "GB/s",
                "note": "a rank could not pin its host pools; no whole-job end-to-end number"}
    ms_all = max_over_ranks(float(ms))
    out = dict(e2e)
    out.update({"value": round(step_bytes(a) * world / (ms_all / 1e3) / 1e9, 2),
                "ms_per_step": round(ms_all, 3),
                "sessions_per_s": round(a.sessions * world / (ms_all / 1e3), 2),
                "h2d_bytes_per_step": e2e["h2d_bytes_per_step"] * world,
                "d2h_bytes_per_step": e2e["d2h_bytes_per_step"] * world,
                "ranks": world, "rank0_value": e2e["value"]})
    return out


def run_e2e(a, ctx, kv, dst, stream, dev):
    """End to end through the library with the state in host memory: each
    step checkpoints every session from K and V page pools that live in
    pinned host memory (the caller hands the library host pointers; its
    kernels read the pages over the host link, pack the records into HBM and
    fingerprint them), restores the records verified into the freshly
    permuted pool in HBM, and copies the session fingerprints to the host.
    Prepared calls (planned once, then launches only) on two streams with two
    sets of records used in turn: step i+1's checkpoint reads the host link
    while step i's restore runs in HBM; the library orders each record's
    rewrite after its last read.  Host -> device: every payload byte, once per
    step; device -> host: one 8-byte session fingerprint per session."""
    from paper_2607_21686_gb300 import pcs

    S = a.sessions
    nb = kv.k_pool.numel() * kv.k_pool.element_size()
    verify = 0 if a.no_verify else 2
    dst_arr = ctx.session_array(dst)
    s_in = torch.cuda.Stream(device=dev)
    s_out = torch.cuda.Stream(device=dev)
    fps_d = torch.empty(2, S, dtype=torch.int64, device=dev)
    fps_h = torch.empty(2, S, dtype=torch.int64, pin_memory=True)
    probes = {}

    class Pipeline:
        """Two record sets, each a prepared checkpoint from the host pools
        and a prepared restore into the HBM pool."""

        def __init__(self, kh, vh):
            arr = ctx.session_array([pcs.kv_session(s, kv.meta[s], kh, vh, kv.page_table[s],
                                                    kv.ring_start[s], a.window)
                                     for s in range(S)])
            self.sets = []
            for _ in range(2):
                cp, hs = ctx.plan_checkpoint(arr, S, stream=s_in)
                rp = ctx.plan_restore(hs, S, dst_arr, verify=verify)
                self.sets.append((cp, rp, hs))
            self.arr = arr

        def step(self, i):
            cp, rp, hs = self.sets[i % 2]
            ctx.plan_run(cp, stream=s_in)
            ctx.plan_run(rp, stream=s_out)
            f = fps_d[i % 2]
            for k in range(S):
                ctx.copy_out(pcs.Snapshot(ctx, hs[k]), 24, 8, f[k:k + 1], stream=s_out)
            with torch.cuda.stream(s_out):
                fps_h[i % 2].copy_(f, non_blocking=True)

        def run(self, n):
            s_in.wait_stream(stream)
            s_out.wait_stream(stream)
            for i in range(n):
                self.step(i)
            stream.wait_stream(s_in)
            stream.wait_stream(s_out)

        def close(self):
            for cp, rp, hs in self.sets:
                ctx.plan_destroy(rp)
                ctx.plan_destroy(cp)
                ctx.delete_raw(hs, S)
            self.sets = []

    def probe(name, kh, vh):
        # Two steps from these host pools: how the pages were pinned shows at
        # this size.
        kh.copy_(kv.k_pool)
        vh.copy_(kv.v_pool)
        pipe = Pipeline(kh, vh)
        pipe.run(2)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        pipe.run(2)
        e1.record(stream)
        torch.cuda.synchronize()
        probes[name] = round(2 * 2 * nb / (e0.elapsed_time(e1) / 1e3) / 1e9, 1)
        return probes[name], pipe

    host, pipe, pinning, rate = [], None, None, 0.0
    huge0 = _anon_huge_bytes()
    try:
        host = [HostBuffer(nb), HostBuffer(nb)]
        kh = host[0].view(kv.k_pool.shape, kv.k_pool.dtype)
        vh = host[1].view(kv.v_pool.shape, kv.v_pool.dtype)
        pinning = "huge-page mapping, cudaHostRegister"
        probes["huge_pages_GiB"] = round((_anon_huge_bytes() - huge0) / 2**30, 1)
        rate, pipe = probe("mapping_GBs_of_pools", kh, vh)
    except Exception:
        if pipe is not None:
            pipe.close()
        for h in host:
            h.close()
        host, pipe, rate = [], None, 0.0
    if rate < 150.0:
        # Without huge pages the host's address translation can slow the link
        # down; the driver's own pinned allocation may do better.  Keep the faster.
        try:
            kt = torch.empty(kv.k_pool.shape, dtype=kv.k_pool.dtype, pin_memory=True)
            vt = torch.empty(kv.v_pool.shape, dtype=kv.v_pool.dtype, pin_memory=True)
            r2, pipe2 = probe("cudaHostAlloc_GBs_of_pools", kt, vt)
            if r2 > rate:
                if pipe is not None:
                    pipe.close()
                for h in host:
                    h.close()
                host, pipe, pinning, rate = [], pipe2, "cudaHostAlloc", r2
            else:
                pipe2.close()
                del kt, vt
        except Exception as ex:  # pinned memory could not be had
            if pipe is None:
                return {"value": None, "unit": "GB/s", "note": "pinned allocation failed: %s" % ex}
    pipe.run(max(1, a.warmup))
    torch.cuda.synchronize()
    ctx.sync()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    pipe.run(a.steps)
    e1.record(stream)
    torch.cuda.synchronize()
    ctx.sync()  # raises if a verified restore found a mismatch
    ms = e0.elapsed_time(e1) / a.steps
    # The fingerprints read back equal the records' session fps.
    last = (a.steps - 1) % 2
    expect = []
    for k in range(S):
        v = ctx.info(pcs.Snapshot(ctx, pipe.sets[last][2][k])).session_fp
        expect.append(v - (1 << 64) if v >= (1 << 63) else v)
    fps_ok = fps_h[last].tolist() == expect
    pipe.close()
    for h in host:
        h.close()
    return {"value": round(step_bytes(a) / (ms / 1e3) / 1e9, 2), "unit": "GB/s",
            "h2d_bytes_per_step": 2 * nb, "d2h_bytes_per_step": S * 8,
            "ms_per_step": round(ms, 3), "sessions_per_s": round(S / (ms / 1e3), 2),
            "steps": a.steps,
            "how": "prepared pcs_checkpoint of the sessions from K/V page pools in pinned host "
                   "memory (the library reads them over the host link) and verified prepared "
                   "pcs_restore into HBM, two record sets on two streams; session fingerprints "
                   "copied to the host every step",
            "h2d_GBs_in_run": round(2 * nb / (ms / 1e3) / 1e9, 1), "fps_read_back_match": fps_ok,
            "pinned": pinning, "pinned_probes": probes}


def measure_suspend_resume(a, ctx, src, dst, stream, dev, groups: int = 8,
                           steps: int | None = None):
    """The KV population crossing the host link both ways every step: suspend
    every session to pinned host memory (checkpoint with
    PCS_PLACE_PINNED_HOST: the library's kernels pack HBM into host records,
    fingerprints fused) and resume it from there (verified restore from the
    host records into the freshly permuted pool in HBM).  The sessions go in
    `groups` groups, each a prepared checkpoint on one stream and a prepared
    restore on another: group g resumes while group g + 1 is suspended, so
    the link carries both directions at once (a call that only crosses the
    link takes half the SMs, so the two kernels can run side by side).
    The library orders every record's rewrite after its last read.  Bytes
    over the link per step: every record written to the host, and read back."""
    from paper_2607_21686_gb300 import pcs

    S = a.sessions
    G = max(1, min(groups, S))
    steps = a.steps if steps is None else steps
    bounds = [S * g // G for g in range(G + 1)]
    verify = 0 if a.no_verify else 2
    cplans, rplans, handles, rec_bytes = [], [], [], 0
    for g in range(G):
        lo, hi = bounds[g], bounds[g + 1]
        cp, hs = ctx.plan_checkpoint(ctx.session_array(src[lo:hi]), hi - lo,
                                     pcs.PCS_PLACE_PINNED_HOST, stream=stream)
        rplans.append(ctx.plan_restore(hs, hi - lo, ctx.session_array(dst[lo:hi]), verify=verify))
        cplans.append(cp)
        handles.append((hs, hi - lo))
        rec_bytes += sum(ctx.info(pcs.Snapshot(ctx, hs[i])).total_bytes for i in range(hi - lo))
    s_out = torch.cuda.Stream(device=dev)
    s_in = torch.cuda.Stream(device=dev)
    suspended = [torch.cuda.Event() for _ in range(G)]

    def run(n):
        s_out.wait_stream(stream)
        s_in.wait_stream(stream)
        for _ in range(n):
            for g in range(G):
                ctx.plan_run(cplans[g], stream=s_out)
                suspended[g].record(s_out)
                s_in.wait_event(suspended[g])
                ctx.plan_run(rplans[g], stream=s_in)
        stream.wait_stream(s_out)
        stream.wait_stream(s_in)

    probe = measure_link(dev, stream)
    run(max(1, a.warmup))
    torch.cuda.synchronize()
    ctx.sync()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    run(steps)
    e1.record(stream)
    torch.cuda.synchronize()
    ctx.sync()  # raises if a verified resume found a mismatch
    ms = e0.elapsed_time(e1) / steps
    # The step's result as the host sees it: every session fingerprint, read
    # from the records in host memory.
    fps = [ctx.info(pcs.Snapshot(ctx, hs[i])).session_fp for hs, n in handles for i in range(n)]
    for p in rplans + cplans:
        ctx.plan_destroy(p)
    for hs, n in handles:
        ctx.delete_raw(hs, n)
    link = rec_bytes / (ms / 1e3) / 1e9
    return {"value": round(step_bytes(a) / (ms / 1e3) / 1e9, 2), "unit": "GB/s",
            "h2d_bytes_per_step": rec_bytes, "d2h_bytes_per_step": rec_bytes,
            "ms_per_step": round(ms, 3), "sessions_per_s": round(S / (ms / 1e3), 2),
            "steps": steps, "groups": G,
            "how": "suspend to pinned host (pcs_checkpoint, PCS_PLACE_PINNED_HOST) + verified "
                   "resume into HBM (pcs_restore from the host records), prepared calls, "
                   "%d groups on two streams" % G,
            "link_GBs_each_way": round(link, 1), "host_link": probe,
            "frac_of_duplex_link": round(link / probe["duplex_GBs_each_way"], 4),
            "session_fps_read": len(fps)}


def main():
    a = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        backend = "nccl" if a.impl == "pcs" else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group(backend=backend)

    if a.impl == "reference":
        line = run_reference(a, rank, world)
        if rank == 0:
            print(json.dumps(line), flush=True)
        if world > 1:
            torch.distributed.destroy_process_group()
        return

    r = run_pcs(a, rank, world, local_rank)
    if rank == 0:
        peaks = load_peaks()
        bytes_step = step_bytes(a) * world
        ms_step = r["ms"] / a.steps
        gbs = bytes_step / (ms_step / 1e3) / 1e9
        sps = a.sessions * world / (ms_step / 1e3)
        # Roofline of the dominant kernel: pack or restore stream pass.
        kt = r["ktimes"]
        cand = {k: v for k, v in kt.items() if k.startswith(("k_stream", "k_bulk"))}
        top = max(cand, key=lambda k: cand[k][1]) if cand else None
        # One pass moves every payload byte once in and once out.
        roof = None
        if top:
            n_l, tot = cand[top]
            per_launch_ms = tot / n_l
            algo = step_bytes(a) // 2     # one pass: read + write of every payload byte
            achieved = algo / (per_launch_ms / 1e3) / 1e9
            roof = {"bound": "hbm", "kernel": top, "achieved": round(achieved, 1),
                    "peak": peaks["hbm_gbs"], "peak_source": peaks["source"], "unit": "GB/s",
                    "frac": round(achieved / peaks["hbm_gbs"], 4),
                    "bytes_per_launch": algo, "ms_per_launch": round(per_launch_ms, 4),
                    "traffic": ncu_traffic(top, a.sessions)}
        cpu = None
        if not a.no_cpu_baseline:
            one = cpu_oracle_rate(a, a.cpu_seconds)
            pool = oracle_pool(host_cores())
            try:
                cpu = cpu_oracle_rate(a, a.cpu_seconds, pool)
            finally:
                if pool is not None:
                    pool.close()
                    pool.join()
            cpu["one_core"] = {k: one[k] for k in ("value", "sessions_per_s", "sample")}
        line = {"metric": METRIC, "value": round(gbs, 2), "unit": "GB/s", "n_gpus": world,
                "steps": a.steps, "warmup": a.warmup, "ms_per_step": round(ms_step, 4),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u64",
                "data": "synthetic",
                "config": bench_config(a, world), "host_cpus": r["host_cpus"],
                "sessions_per_s": round(sps, 2),
                "frac_of_nominal_8tbs": round(gbs / 8000.0, 4),
                "roofline": roof, "cpu_baseline": cpu, "e2e": r["e2e"],
                "gpu_launches": r["launches"], "clocks": r["clocks"], "rows": r["rows"],
                "kernel_ms": {k: [v[0], round(v[1], 3)] for k, v in r["ktimes"].items()}}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
