"""GPU parity at the limits: sessions of thousands of sections and a buffer
past 4 GiB (offsets and chunk counts beyond 32 bits of bytes).

Records equal the oracle's byte for byte; restored bytes equal the live ones.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs
from helpers import np_bytes

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("n_sections", [70, 2048, 2049, 5000])
def test_many_sections_in_one_session(ctx, dev, n_sections):
    # Sizes from 0 to 9 KiB, many not multiples of 16, so the small-call,
    # fused and split finalisation paths all see odd payloads.
    rnd = np.random.default_rng(n_sections)
    sizes = rnd.integers(0, 9 * 1024, n_sections)
    sizes[::13] = 0
    host = [rnd.integers(0, 256, int(n), dtype=np.uint8) for n in sizes]
    bufs = [torch.from_numpy(h).to(dev) for h in host]
    secs = [pcs.contig_section(pcs.PCS_SEC_OBS, b, dim0=b.numel()) for b in bufs]
    sess = pcs.Session(9, pcs.PCS_KIND_MARKOV, secs, keep=bufs)
    snap = ctx.checkpoint([sess])[0]
    spec = oracle.SessionSpec(9, oracle.KIND_MARKOV)
    for h in host:
        spec.contig(oracle.SEC_OBS, oracle.DT_U8, h, dim0=h.size)
    ref = oracle.pack(spec)
    assert np.array_equal(ctx.record(snap).numpy(), ref)
    outs = [torch.full_like(b, 7) for b in bufs]
    ctx.restore([snap], [pcs.Session(9, pcs.PCS_KIND_MARKOV,
                                     [pcs.contig_section(pcs.PCS_SEC_OBS, o, dim0=o.numel())
                                      for o in outs], keep=outs)], verify=True)
    torch.cuda.synchronize()
    assert all(torch.equal(o, b) for o, b in zip(outs, bufs))
    ctx.delete(snap)


@pytest.mark.slow
def test_buffer_past_4_gib(ctx, dev):
    # 4.5 GiB + 13 bytes: more than 2^32 bytes and 2^20 chunks, ragged tail.
    n = (9 << 29) + 13
    g = torch.Generator(device=dev).manual_seed(45)
    x = torch.randint(0, 256, (n,), generator=g, device=dev, dtype=torch.uint8)
    fp = int(ctx.fingerprint([x])[0])
    hx = np_bytes(x)
    assert fp & (2**64 - 1) == oracle.fingerprint(hx)
    # The same bytes through a record and back into another buffer.
    snap = ctx.checkpoint([pcs.Session(1, pcs.PCS_KIND_MARKOV,
                                       [pcs.contig_section(pcs.PCS_SEC_OBS, x, dim0=n)],
                                       keep=[x])])[0]
    assert ctx.section(snap, 0).fp == oracle.fingerprint(hx)
    del hx
    y = torch.zeros_like(x)
    ctx.restore([snap], [pcs.Session(1, pcs.PCS_KIND_MARKOV,
                                     [pcs.contig_section(pcs.PCS_SEC_OBS, y, dim0=n)],
                                     keep=[y])], verify=True)
    torch.cuda.synchronize()
    assert torch.equal(x, y)
    ctx.delete(snap)
