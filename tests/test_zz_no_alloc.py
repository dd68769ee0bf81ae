"""pcs_fingerprint_static, the allocation-free entry point, against pcs_fingerprint.

Some callers of this library cannot allocate device memory: a serving
process that has already reserved nearly all of HBM for its own page pools,
or a latency-critical loop that cannot pay for the synchronisation cudaMalloc
and cudaFree bring.  For them pcs_fingerprint_static computes the same
fingerprints with no context and no allocation, using one fixed device array
as its only working memory.

This test calls it through the C ABI twice in a row on different inputs and
checks every result against the context-based pcs_fingerprint (the results
are integers, so they must be equal bit for bit).  It sits in a file that
pytest collects last and must pass both on its own in a fresh process and
after the other tests.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs
from helpers import np_bytes, u64

pytestmark = pytest.mark.gpu


def _bufs(tensors):
    arr = (pcs.pcs_buf * max(len(tensors), 1))()
    for i, t in enumerate(tensors):
        arr[i] = pcs.pcs_buf(ptr=t.data_ptr() if t.numel() else None,
                             bytes=t.numel() * t.element_size(), dtype=0, flags=0)
    return arr


def _static(lib, tensors, out):
    stream = torch.cuda.current_stream().cuda_stream
    return lib.pcs_fingerprint_static(_bufs(tensors), len(tensors),
                                      out.data_ptr() if out.numel() else None, stream)


def _inputs(seed, sizes, dev):
    g = torch.Generator().manual_seed(seed)
    out = []
    for n in sizes:
        t = torch.randint(0, 256, (n + 3,), generator=g, dtype=torch.uint8).to(dev)
        out.append(t[:n])
        out.append(t[3:3 + n])  # an unaligned view of the same length
    return out


def test_static_matches_context_twice(ctx, dev):
    lib = pcs.load_library()
    first = _inputs(1, [0, 1, 17, 4096, 4097, 3 * 4096 + 5, 1 << 20, (5 << 20) + 3], dev)
    second = _inputs(2, [16384 * 7, 100, (3 << 20) + 48, 65 * 4096 + 4095, 8], dev)
    for tensors in (first, second):
        out = torch.full((len(tensors),), -1, dtype=torch.int64, device=dev)
        assert _static(lib, tensors, out) == pcs.PCS_OK, lib.pcs_last_error()
        want = ctx.fingerprint(tensors)
        torch.cuda.synchronize()
        assert u64(out) == u64(want)
    # And against the oracle for the last call.
    assert u64(out) == [oracle.fingerprint(np_bytes(t)) for t in second]


def _task_log2(sizes):
    """2^g chunks per warp task, as the entry point picks it: the smallest g
    whose tasks fit the fixed node array and leave fewer than 2 x 8192 tasks'
    worth of chunks per doubling (a larger call takes larger tasks)."""
    chunks = [max(1, -(-n // 4096)) for n in sizes]
    g = 0
    while g < 5 and (sum(-(-c // (1 << g)) for c in chunks) > pcs.PCS_STATIC_MAX_NODES
                     or (sum(chunks) >> (g + 1)) >= 8192):
        g += 1
    return g


# Totals from about 100 MiB to 1.3 GiB: one case per task size 2^1 .. 2^5
# chunks, chunk counts not multiples of 2^g, with empty and unaligned views.
_LARGE = {
    1: [(60 << 20) + 4097, (40 << 20) + 3, 0],
    2: [(150 << 20) + 12345, 7, (50 << 20) + 4096 * 3 + 1],
    3: [(300 << 20) + 4096 * 5 + 9, 0, (100 << 20) + 1],
    4: [(500 << 20) + 4096 * 13 + 5, (200 << 20) + 4096 * 7],
    5: [(900 << 20) + 4096 * 29 + 11, 4095, (400 << 20) + 4096 * 31 + 3],
}


@pytest.mark.parametrize("g", sorted(_LARGE))
def test_static_large_task_groups(ctx, dev, g):
    # Every call past 64 MiB groups 2^g chunks per warp task: the per-warp
    # loop over the group, the lane that keeps each chunk's hash and the
    # warp tree over a partial last group.
    sizes = _LARGE[g]
    assert _task_log2(sizes) == g
    lib = pcs.load_library()
    gen = torch.Generator(device=dev).manual_seed(100 + g)
    tensors = []
    for i, n in enumerate(sizes):
        t = torch.randint(0, 256, (n + 3,), generator=gen, dtype=torch.uint8, device=dev)
        tensors.append(t[3:] if i % 2 else t[:n])  # odd buffers: views off a 16-byte boundary
    for _ in range(2):
        out = torch.full((len(tensors),), -1, dtype=torch.int64, device=dev)
        assert _static(lib, tensors, out) == pcs.PCS_OK, lib.pcs_last_error()
        want = ctx.fingerprint(tensors)
        torch.cuda.synchronize()
        assert u64(out) == u64(want)
    assert u64(out) == [oracle.fingerprint(np_bytes(t)) for t in tensors]


def test_static_limits_are_rejected_before_any_work(dev):
    lib = pcs.load_library()
    t = torch.zeros(16, dtype=torch.uint8, device=dev)
    out = torch.zeros(pcs.PCS_STATIC_MAX_BUFFERS + 1, dtype=torch.int64, device=dev)
    too_many = [t] * (pcs.PCS_STATIC_MAX_BUFFERS + 1)
    assert _static(lib, too_many, out) == pcs.PCS_E_INVAL
    assert b"64" in lib.pcs_last_error()
    # A description far beyond the fixed scratch is refused on the host; the
    # buffer is never read.
    arr = (pcs.pcs_buf * 1)()
    arr[0] = pcs.pcs_buf(ptr=t.data_ptr(), bytes=1 << 40, dtype=0, flags=0)
    st = lib.pcs_fingerprint_static(arr, 1, out.data_ptr(),
                                    torch.cuda.current_stream().cuda_stream)
    assert st == pcs.PCS_E_INVAL
    assert b"scratch" in lib.pcs_last_error()
    assert lib.pcs_fingerprint_static(arr, 0, None, None) == pcs.PCS_OK
