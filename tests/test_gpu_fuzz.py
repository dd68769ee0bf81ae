"""GPU: seeded random sessions against the oracle.

Each trial draws sessions of one to six sections with random layouts --
contiguous buffers of random length at random byte offsets (16-byte, 4-byte
and 1-byte aligned, empty ones too), rows of random size gathered by random
(repeating) indices, and paged rings of random window, page size and start
over a randomly permuted pool -- packs them in one call, compares every record
with the oracle's byte for byte, restores them verified into fresh targets
(rows into contiguous buffers, rings into a freshly permuted pool at the
stored ring start) and compares every restored byte with the source.  Sizes
are drawn around 4 KiB chunk and 8 KiB tile boundaries so that tails,
padding and the split loads meet every case; the calls range from one fused
launch to the TMA kernels."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs

pytestmark = pytest.mark.gpu

def _size(rnd, big):
    base = int(rnd.choice([0, 1, 2, 5, 40, 100, 300] if not big else [64, 128, 256, 700]))
    return max(0, base * 8192 + int(rnd.integers(-48, 49)) * int(rnd.choice([1, 16])))


def _draw_session(rnd, dev, big):
    """One random session: (GPU sections, oracle spec builder, restore plan)."""
    secs, keep, parts = [], [], []
    for _ in range(int(rnd.integers(1, 7))):
        kind = rnd.choice(["contig", "rows", "ring"], p=[0.5, 0.25, 0.25])
        if kind == "contig":
            n = _size(rnd, big)
            off = int(rnd.choice([0, 16, 4, 1]))
            t = torch.randint(0, 256, (n + off + 16,), dtype=torch.uint8, device=dev)
            v = t[off:off + n]
            secs.append(pcs.contig_section(pcs.PCS_SEC_OBS, v))
            keep.append(t)
            parts.append(("contig", v))
        elif kind == "rows":
            rb = int(rnd.choice([16, 48, 512, 1040, 2048, 32768]))
            rows = int(rnd.integers(1, 160))
            k = int(rnd.integers(0, 2 * rows))
            base = torch.randint(0, 256, (rows, rb), dtype=torch.uint8, device=dev)
            idx = torch.from_numpy(rnd.integers(0, rows, k).astype(np.int32)).to(dev)
            secs.append(pcs.rows_section(pcs.PCS_SEC_VALUES, base, idx))
            keep += [base, idx]
            parts.append(("rows", base, idx))
        else:
            pr = 16
            rb = int(rnd.choice([512, 2048]))
            window = int(rnd.choice([16, 64, 256, 1024]))
            pages = window // pr
            pool_pages = 2 * pages + 3
            pool = torch.randint(0, 256, (pool_pages, pr, rb), dtype=torch.uint8, device=dev)
            pt = torch.from_numpy(rnd.permutation(pool_pages)[:pages].astype(np.int32)).to(dev)
            start = int(rnd.integers(0, window))
            secs.append(pcs.ring_section(pcs.PCS_SEC_K, pool, pt, start, window))
            keep += [pool, pt]
            parts.append(("ring", pool, pt, start, window))
    return secs, keep, parts


def _logical(part):
    """The section's bytes in logical order, on the host."""
    if part[0] == "contig":
        return part[1].cpu().numpy()
    if part[0] == "rows":
        return part[1].cpu().numpy()[part[2].cpu().numpy().astype(np.int64)].reshape(-1)
    _, pool, pt, start, window = part
    pr = pool.shape[1]
    slot = (start + np.arange(window)) % window
    p = pool.cpu().numpy()
    return p[pt.cpu().numpy()[slot // pr], slot % pr].reshape(-1)


def _oracle_spec(sid, parts):
    sp = oracle.SessionSpec(sid, oracle.KIND_MARKOV)
    for part in parts:
        if part[0] == "contig":
            sp.contig(pcs.PCS_SEC_OBS, oracle.DT_U8, np.ascontiguousarray(part[1].cpu().numpy()))
        elif part[0] == "rows":
            base = np.ascontiguousarray(part[1].cpu().numpy())
            idx = np.ascontiguousarray(part[2].cpu().numpy())
            sp.rows(pcs.PCS_SEC_VALUES, oracle.DT_U8, base, base.shape[1], idx,
                    dim0=idx.size, dim1=base.shape[1])
        else:
            _, pool, pt, start, window = part
            p = np.ascontiguousarray(pool.cpu().numpy())
            sp.ring(pcs.PCS_SEC_K, oracle.DT_U8, p, p.shape[2],
                    np.ascontiguousarray(pt.cpu().numpy()), start, window, p.shape[1],
                    dim0=window, dim1=p.shape[2])
    return sp


@pytest.mark.parametrize("trial", range(24))
def test_random_sessions_round_trip(ctx, dev, trial):
    rnd = np.random.default_rng(4100 + trial)
    torch.manual_seed(4100 + trial)
    big = trial % 2 == 1
    n = int(rnd.integers(1, 24 if not big else 10))
    drawn = [_draw_session(rnd, dev, big) for _ in range(n)]
    sessions = [pcs.Session(s, pcs.PCS_KIND_MARKOV, secs, keep)
                for s, (secs, keep, _) in enumerate(drawn)]
    placement = pcs.PCS_PLACE_PINNED_HOST if trial % 4 == 3 else pcs.PCS_PLACE_DEVICE
    snaps = ctx.checkpoint(sessions, placement=placement)
    for s, (_, _, parts) in enumerate(drawn):
        ref = oracle.pack(_oracle_spec(s, parts))
        assert np.array_equal(ctx.record(snaps[s]).numpy(), ref), (trial, s)
    # Verified restore into fresh targets: rows into contiguous buffers,
    # rings into a freshly permuted pool at the stored start.
    targets, outs = [], []
    for s, (_, _, parts) in enumerate(drawn):
        tsecs, tkeep, tparts = [], [], []
        for part in parts:
            if part[0] == "ring":
                _, pool, pt, start, window = part
                pool2 = torch.zeros_like(pool)
                pt2 = torch.from_numpy(rnd.permutation(pool.shape[0])[:pt.numel()]
                                       .astype(np.int32)).to(dev)
                tsecs.append(pcs.ring_section(pcs.PCS_SEC_K, pool2, pt2,
                                              pcs.PCS_RING_START_FROM_SNAPSHOT, window))
                tkeep += [pool2, pt2]
                tparts.append(("ring", pool2, pt2, start, window))
            else:
                n_bytes = _logical(part).size
                off = int(rnd.choice([0, 16, 4, 1]))
                t = torch.zeros(n_bytes + off + 16, dtype=torch.uint8, device=dev)
                v = t[off:off + n_bytes]
                tsecs.append(pcs.contig_section(pcs.PCS_SEC_OBS, v))
                tkeep.append(t)
                tparts.append(("contig", v))
        targets.append(pcs.Session(s, pcs.PCS_KIND_MARKOV, tsecs, tkeep))
        outs.append(tparts)
    ctx.restore(snaps, targets, verify=True)
    torch.cuda.synchronize()
    for s, (_, _, parts) in enumerate(drawn):
        for j, (a, b) in enumerate(zip(parts, outs[s])):
            assert np.array_equal(_logical(a), _logical(b)), (trial, s, j)
    for x in snaps:
        ctx.delete(x)
