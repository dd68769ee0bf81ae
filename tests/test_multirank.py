"""The multi-rank paths on CPU with gloo (world size 2).

Sessions are independent, so ranks share nothing on the data path of the
step; bench.py's only exchange is the max over ranks of the timed region.
The one real exchange of the method is the host budget of banks sharded
across ranks (Sec. 7.5: every bank keeps the same fraction B / T of the whole
population): one all-reduced scalar, T.  These tests exercise both
reductions and the launch contract of the reference arm under torchrun.
"""
import json
import os
import subprocess
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    import bench
    out[rank] = bench.max_over_ranks(10.0 + 5.0 * rank)
    torch.distributed.destroy_process_group()


def _e2e_worker(rank, world, port, out, fail_rank):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    import bench

    class A:
        sessions, layers, heads, head_dim, window, page_rows = 256, 24, 16, 64, 1024, 16
    if rank == fail_rank:
        mine = {"value": None, "unit": "GB/s", "note": "pinned allocation failed"}
    else:
        ms = 120.0 + 10.0 * rank
        mine = {"value": round(bench.step_bytes(A) / (ms / 1e3) / 1e9, 2), "unit": "GB/s",
                "ms_per_step": ms, "h2d_bytes_per_step": 100, "d2h_bytes_per_step": 8}
    out[rank] = bench.e2e_over_ranks(A, mine, world)
    torch.distributed.destroy_process_group()


def _budget_worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    from paper_2607_21686_gb300 import pcs
    import numpy as np
    rnd = np.random.default_rng(5)
    n = rnd.integers(256, 4097, 2048)
    E = rnd.choice([3072, 1024, 5000], 2048)
    mine = range(rank, 2048, world)  # interleaved shards
    banks = (pcs.pcs_bank * len(mine))()
    for j, s in enumerate(mine):
        banks[j] = pcs.pcs_bank(n_entries=int(n[s]), key_dim=8, key_dtype=pcs.PCS_DT_F16,
                                entry_bytes=int(E[s]))
    t_local = int(sum(int(n[s]) * int(E[s]) for s in mine))
    t = torch.tensor([t_local], dtype=torch.int64)
    torch.distributed.all_reduce(t)  # the one scalar the budget rule needs
    p = pcs.Context.params(pcs.PCS_K_BUDGET, budget=8 << 30, total_bytes=int(t.item()))
    out[rank] = dict(zip(mine, pcs.Context.prune_counts(banks, len(mine), p)))
    torch.distributed.destroy_process_group()


def _free_port():
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def test_max_over_ranks_gloo():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        assert dict(out) == {0: 15.0, 1: 15.0}


def test_reference_arm_under_torchrun():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0",
           "--cpu-seconds", "1", "--layers", "2"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["e2e"]["h2d_bytes_per_step"] == 0


def test_sharded_budget_matches_one_process():
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        procs = [ctx.Process(target=_budget_worker, args=(r, 2, port, out)) for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        k = {**out[0], **out[1]}
    import numpy as np
    import oracle
    rnd = np.random.default_rng(5)
    n = rnd.integers(256, 4097, 2048)
    E = rnd.choice([3072, 1024, 5000], 2048)
    want = oracle.k_budget(n, E.astype(np.uint64), 8 << 30)
    assert [k[s] for s in range(2048)] == want.tolist()


@pytest.mark.parametrize("fail_rank", [-1, 1])
def test_e2e_over_ranks_gloo(fail_rank):
    """The whole-job end-to-end line: both ranks' step bytes over the slower
    rank's time; no number at all when a rank could not run its end to end."""
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        procs = [ctx.Process(target=_e2e_worker, args=(r, 2, port, out, fail_rank))
                 for r in range(2)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = {r: {k: v for k, v in d.items() if k != "rank0_value"} for r, d in dict(out).items()}
    assert res[0] == res[1]
    if fail_rank >= 0:
        assert res[0]["value"] is None
    else:
        step = 4 * 256 * (2 * 24 * 1024 * 16 * 64 * 2 + 32)
        assert res[0]["ms_per_step"] == 130.0
        assert res[0]["value"] == round(2 * step / 0.130 / 1e9, 2)
        assert res[0]["h2d_bytes_per_step"] == 200 and res[0]["ranks"] == 2
