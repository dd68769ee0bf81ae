"""GPU: durability across processes and an out-of-memory path.

I2 in its strongest form (Sec. 7.2, "Across a process boundary"): one
process checkpoints a session, writes the record to a file and dies without
cleaning up; a fresh process reads the file and restores the exact bytes.
An arena cap makes allocation failure happen on purpose: the call fails with
PCS_E_NOMEM before any launch, leaves nothing behind, and succeeds once
memory is free again.
"""
import os
import subprocess
import sys

import pytest
import torch

from paper_2607_21686_gb300 import pcs

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_WRITER = r"""
import os, sys, torch
sys.path.insert(0, sys.argv[1])
from paper_2607_21686_gb300 import pcs, synth
m = synth.markov(seed=4242)
ctx = pcs.Context(0)
obs, rng = m.obs.cuda(), m.rng.cuda()
snap = ctx.checkpoint([pcs.markov_session(8, obs, rng)])[0]
ctx.write_file(snap, sys.argv[2])
print("fp", ctx.info(snap).session_fp, flush=True)
os._exit(0)   # die: no context teardown, no frees
"""

_READER = r"""
import sys, torch
sys.path.insert(0, sys.argv[1])
from paper_2607_21686_gb300 import pcs, synth
m = synth.markov(seed=4242)
ctx = pcs.Context(0)
snap = ctx.read_file(sys.argv[2])
o, r = torch.zeros_like(m.obs).cuda(), torch.zeros_like(m.rng).cuda()
ctx.restore([snap], [pcs.markov_session(8, o, r)], verify=True)
torch.cuda.synchronize()
assert torch.equal(o.cpu(), m.obs) and torch.equal(r.cpu(), m.rng)
print("fp", ctx.info(snap).session_fp, flush=True)
"""


def test_record_survives_process_death(tmp_path):
    path = str(tmp_path / "dead.pcs")
    w = subprocess.run([sys.executable, "-c", _WRITER, ROOT, path], capture_output=True,
                       text=True, timeout=300)
    assert w.returncode == 0, w.stderr[-2000:]
    r = subprocess.run([sys.executable, "-c", _READER, ROOT, path], capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    fp_w = [l for l in w.stdout.splitlines() if l.startswith("fp")]
    fp_r = [l for l in r.stdout.splitlines() if l.startswith("fp")]
    assert fp_w and fp_w == fp_r


def test_arena_cap_gives_nomem_then_recovers(dev):
    with pcs.Context(0) as c:
        c.set_arena_limit(pcs.PCS_PLACE_DEVICE, 300 << 20)
        x = torch.randint(0, 256, (200 << 20,), device=dev, dtype=torch.uint8)
        y = torch.randint(0, 256, (200 << 20,), device=dev, dtype=torch.uint8)

        def sess(t):
            return pcs.Session(1, pcs.PCS_KIND_MARKOV,
                               [pcs.contig_section(pcs.PCS_SEC_OBS, t, dim0=t.numel())], keep=[t])
        a = c.checkpoint([sess(x)])[0]
        live = c.stats().live_snapshots
        with pytest.raises(pcs.PcsError) as e:
            c.checkpoint([sess(y)])
        assert e.value.status == pcs.PCS_E_NOMEM
        assert c.stats().live_snapshots == live
        c.delete(a)
        b = c.checkpoint([sess(y)])[0]       # the freed range is enough again
        c.sync()
        z = torch.zeros_like(y)
        c.restore([b], [sess(z)], verify=True)
        torch.cuda.synchronize()
        assert torch.equal(z, y)
        c.delete(b)
        c.set_arena_limit(pcs.PCS_PLACE_DEVICE, 0)
