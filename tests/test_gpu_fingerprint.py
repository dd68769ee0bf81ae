"""GPU parity: fingerprint and classify through the C ABI vs the oracle.

Bit-exact: every fingerprint and every must-snapshot flag (Sec. 4
FINGERPRINT step 1 at epsilon = 0; Sec. 3 "The partition").
"""
import ctypes

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_bytes, u64

pytestmark = pytest.mark.gpu

EDGE_SIZES = [0, 1, 7, 15, 16, 17, 255, 256, 4095, 4096, 4097, 8192, 3 * 4096 + 5,
              31 * 4096 + 100, 32 * 4096, 33 * 4096 + 1, 64 * 4096, 65 * 4096 + 4095,
              (1 << 20) + 3, (5 << 20) + 4097]


def _rand_bytes(n, seed, dev):
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    return torch.randint(0, 256, (n,), generator=g, dtype=torch.uint8).to(dev)


def test_edge_sizes_bit_exact(ctx, dev):
    bufs = [_rand_bytes(n, 100 + i, dev) for i, n in enumerate(EDGE_SIZES)]
    got = u64(ctx.fingerprint(bufs))
    want = [oracle.fingerprint(np_bytes(b)) for b in bufs]
    assert got == want


def test_result_independent_of_batching(ctx, dev):
    # One buffer alone (small warp tasks) vs inside a large batch (32-chunk
    # tasks): the aligned-group tree makes the result scheduling-free.
    big = [_rand_bytes(8 << 20, 7, dev) for _ in range(8)]
    probe = _rand_bytes(77 * 4096 + 9, 8, dev)
    alone = u64(ctx.fingerprint([probe]))[0]
    batched = u64(ctx.fingerprint(big + [probe]))[-1]
    assert alone == batched == oracle.fingerprint(np_bytes(probe))


def test_dtypes_and_views(ctx, dev):
    g = torch.Generator(device="cpu")
    g.manual_seed(3)
    ts = [torch.randn(1000, generator=g).to(torch.bfloat16), torch.randn(333, generator=g).half(),
          torch.randint(-2**62, 2**62, (77,), generator=g, dtype=torch.int64),
          torch.randn(4096 + 1, generator=g)]
    got = u64(ctx.fingerprint([t.to(dev) for t in ts]))
    assert got == [oracle.fingerprint(np_bytes(t)) for t in ts]


def test_classify_small_sweep(ctx, dev):
    sw = synth.sweep(seed=11, n=60, lo=64, hi=1 << 20)
    before = [t.to(dev) for t in sw.before]
    after = [t.to(dev) for t in sw.after]
    fp0 = ctx.fingerprint(before)
    must, fp1 = ctx.classify(after, fp0)
    want0 = oracle.fingerprint_many([np_bytes(t) for t in sw.before])
    want1 = oracle.fingerprint_many([np_bytes(t) for t in sw.after])
    assert u64(fp0) == [int(x) for x in want0]
    assert u64(fp1) == [int(x) for x in want1]
    flags = must.cpu().numpy().tolist()
    assert flags == oracle.classify(want0, want1).tolist()
    assert flags == [1 if f else 0 for f in sw.flipped]


def test_rng_single_bit_flip(ctx, dev):
    # Wrong-value control (Sec. 4): one flipped RNG bit changes the fp.
    m = synth.markov(seed=5)
    rng = m.rng.to(dev)
    base = u64(ctx.fingerprint([rng]))[0]
    for bit in range(128):
        r2 = rng.clone()
        r2.view(torch.uint8)[bit // 8] ^= (1 << (bit % 8))
        assert u64(ctx.fingerprint([r2]))[0] != base


def test_unaligned_views(ctx, dev):
    # Views at every offset mod 16 (byte and 4-byte aligned paths).
    base = _rand_bytes(3 * 4096 + 200, 9, dev)
    views = [base[o:o + n] for o in [1, 2, 3, 4, 5, 8, 12, 15] for n in [0, 1, 5, 17, 4100]]
    got = u64(ctx.fingerprint(views))
    assert got == [oracle.fingerprint(np_bytes(v)) for v in views]


def test_empty_list(ctx, dev):
    out = ctx.fingerprint([])
    assert out.numel() == 0


@pytest.mark.slow
def test_classify_full_size_sweep(ctx, dev):
    # 200 buffers, 64 B .. 256 MiB log-uniform (about 3.5 GB per pass).
    sw = synth.sweep(device=dev)
    fp0 = ctx.fingerprint(sw.before)
    must, fp1 = ctx.classify(sw.after, fp0)
    torch.cuda.synchronize()
    flags = must.cpu().numpy().tolist()
    # Property that holds at any size: a single-bit change always changes the fp.
    assert flags == [1 if f else 0 for f in sw.flipped]
    # Every output against the oracle, fingerprinted by host threads (the
    # oracle's C calls release the GIL), a batch of buffers at a time.
    got0, got1 = u64(fp0), u64(fp1)
    order = sorted(range(len(sw.sizes)), key=lambda i: -sw.sizes[i])
    with ThreadPoolExecutor(max(1, len(os.sched_getaffinity(0)))) as pool:
        for b0 in range(0, len(order), 16):
            batch = order[b0:b0 + 16]
            host = [(i, np_bytes(sw.before[i]), np_bytes(sw.after[i])) for i in batch]
            futs = [(i, pool.submit(oracle.fingerprint, hb), pool.submit(oracle.fingerprint, ha))
                    for i, hb, ha in host]
            for i, f0, f1 in futs:
                assert got0[i] == f0.result(), i
                assert got1[i] == f1.result(), i
