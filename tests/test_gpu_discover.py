"""GPU parity: the byte-mismatch distance and the state / witness read test.

pcs_mismatch against the oracle's count on pairs of every alignment, length
difference and size (several 16 KiB tiles and ragged tails), and on the
classification sweep's recompute pass (one differing byte exactly where a bit
was flipped).  pcs_classify_reads against the oracle's overlap test on views
of one device tensor (overlapping, nested, empty, adjacent).  Then the whole
Sec. 4 procedure on a small synthetic session model run on the GPU, whose
PCS is known by construction.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_bytes

pytestmark = pytest.mark.gpu


def test_mismatch_matches_oracle(ctx, dev):
    g = torch.Generator().manual_seed(3)
    base_a = torch.randint(0, 256, (300000,), generator=g, dtype=torch.uint8)
    base_b = base_a.clone()
    flip = torch.randint(0, 300000, (5000,), generator=g)
    base_b[flip] ^= torch.randint(1, 256, (5000,), generator=g, dtype=torch.uint8)
    da, db = base_a.to(dev), base_b.to(dev)
    cases = [(0, 0, 0), (0, 0, 1), (0, 0, 16), (0, 0, 16384), (0, 0, 16385), (0, 0, 100000),
             (16, 48, 65536 + 5), (1, 1, 50000), (3, 7, 40000), (5, 5, 17), (0, 0, 250000)]
    a_list, b_list, want = [], [], []
    for oa, ob, n in cases:
        for extra in (0, 9):
            ta, tb = da[oa:oa + n], db[ob:ob + n + extra]
            a_list.append(ta)
            b_list.append(tb)
            want.append(oracle.mismatch(base_a[oa:oa + n].numpy(), base_b[ob:ob + n + extra].numpy()))
    got = ctx.mismatch(a_list, b_list)
    ctx.sync()
    assert got.cpu().tolist() == want


def test_mismatch_on_the_recompute_pass(ctx, dev):
    # Config 4 at a small size: a flipped bit is exactly one differing byte.
    sw = synth.sweep(n=40, hi=4 << 20, device=dev)
    got = ctx.mismatch(sw.before, sw.after).cpu().tolist()
    assert got == [1 if f else 0 for f in sw.flipped]
    for i in (0, 7, 39):
        assert got[i] == oracle.mismatch(np_bytes(sw.before[i]), np_bytes(sw.after[i]))


@pytest.mark.parametrize("seed", range(4))
def test_classify_reads_matches_oracle(ctx, dev, seed):
    rnd = np.random.default_rng(seed)
    space = torch.zeros(1 << 16, dtype=torch.uint8, device=dev)
    base = space.data_ptr()
    bufs, spans = [], []
    for _ in range(300):
        o, n = int(rnd.integers(0, 60000)), int(rnd.integers(0, 3000))
        bufs.append(space[o:o + n])
        spans.append((base + o, n))
    bufs.append(space[100:100])        # empty
    spans.append((base + 100, 0))
    m = 2000
    ro = rnd.integers(0, 65000, m)
    rl = rnd.integers(0, 64, m)
    rl[::7] = 0
    reads = [(base + int(o), int(n)) for o, n in zip(ro, rl)]
    addr = torch.tensor([r[0] for r in reads], dtype=torch.int64, device=dev)
    nb = torch.tensor([r[1] for r in reads], dtype=torch.int64, device=dev)
    got = ctx.classify_reads(bufs, addr, nb)
    ctx.sync()
    assert got.cpu().numpy().tolist() == oracle.classify_reads(spans, reads).tolist()


def test_classify_reads_without_reads(ctx, dev):
    x = torch.zeros(64, dtype=torch.uint8, device=dev)
    e = torch.empty(0, dtype=torch.int64, device=dev)
    assert ctx.classify_reads([x[:8], x[8:]], e, e).cpu().tolist() == [0, 0]


class _Model:
    """A small session model on the GPU.

    Components: obs, rng, cache (= a function of obs, rebuilt on resume),
    frame (the last output: kept for scoring, never read on resume), a and b
    (mirrors of each other: resume uses a if its check word is right, else b).
    """
    names = ["obs", "rng", "cache", "frame", "a", "b"]

    def __init__(self, dev):
        g = torch.Generator(device=dev).manual_seed(11)
        self.obs = torch.randint(0, 256, (3, 64, 64), generator=g, device=dev, dtype=torch.uint8)
        self.rng = torch.randint(0, 2**62, (2,), generator=g, device=dev, dtype=torch.int64)
        self.a = torch.randint(0, 256, (4096,), generator=g, device=dev, dtype=torch.uint8)
        self.a[0] = 0x5A
        self.b = self.a.clone()
        self.cache = self.derive_cache()
        self.frame = self.step()

    def parts(self):
        return [self.obs, self.rng, self.cache, self.frame, self.a, self.b]

    def derive_cache(self):
        return (self.obs.to(torch.int32) * 7 % 251).to(torch.uint8)

    def resume(self):
        self.cache = self.derive_cache()
        reads = [self.obs, self.rng, self.a if int(self.a[0]) == 0x5A else self.b]
        return reads

    def step(self):
        mem = self.a if int(self.a[0]) == 0x5A else self.b
        noise = (self.rng[0] % 251).to(torch.int32)
        out = (self.obs.to(torch.int32) + self.cache.to(torch.int32) + noise) % 256
        return (out.reshape(-1)[:4096] ^ mem.to(torch.int32)).to(torch.uint8)


def test_discovery_on_a_gpu_model(ctx, dev):
    m = _Model(dev)
    sess = [pcs.contig_section(i + 1, t) for i, t in enumerate(m.parts())]
    snap = ctx.checkpoint([pcs.Session(0, pcs.PCS_KIND_MARKOV, sess, keep=m.parts())])[0]
    reference = m.step()
    scratch = [torch.empty_like(t) for t in m.parts()]
    log = []

    def probe(keep):
        # Restore the record into scratch; the kept components come back from
        # it, every byte of the others is left changed (the excursion).
        ctx.restore([snap], [pcs.Session(0, pcs.PCS_KIND_MARKOV,
                                         [pcs.contig_section(i + 1, t)
                                          for i, t in enumerate(scratch)], keep=scratch)])
        for k, t, s in zip(keep, m.parts(), scratch):
            t.copy_(s if k else s ^ (1 if s.dtype == torch.int64 else 0xFF))
        reads = m.resume()
        log.append(reads)
        out = m.step()
        d = int(ctx.mismatch([out], [reference])[0])
        assert d == oracle.mismatch(out.cpu().numpy(), reference.cpu().numpy())
        return d

    flags, probes, ok = pcs.discover(6, probe, 0)
    # obs and rng are necessary; cache is rebuilt; frame is never read; a and
    # b stand in for each other, so the fallback adds the first of them.
    assert dict(zip(_Model.names, flags)) == {"obs": 1, "rng": 1, "cache": 0, "frame": 0,
                                               "a": 1, "b": 0}
    assert ok and probes == 6 + 1 + 4
    # State versus witness on the full restore: resume reads obs, rng and a.
    for t, s in zip(m.parts(), scratch):
        t.copy_(s)
    reads = m.resume()
    addr = torch.tensor([r.data_ptr() for r in reads], dtype=torch.int64, device=dev)
    nb = torch.tensor([r.numel() * r.element_size() for r in reads], dtype=torch.int64, device=dev)
    state = ctx.classify_reads(m.parts(), addr, nb).cpu().tolist()
    assert dict(zip(_Model.names, state)) == {"obs": 1, "rng": 1, "cache": 0, "frame": 0,
                                               "a": 1, "b": 0}
    ctx.delete(snap)
