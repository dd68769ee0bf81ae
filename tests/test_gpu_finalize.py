"""GPU: finalisation of sessions with many sections (more than 32: a warp per
section, then a warp per session) against the oracle, and what a verified
restore of such sessions reports for a flipped payload byte, a flipped stored
section fingerprint and a flipped stored session fingerprint (I1, I4)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs, synth
from helpers import np_view

pytestmark = pytest.mark.gpu


def _kv_setup(dev, sessions=4, layers=24, heads=2, seed=404):
    kv = synth.kv(seed=seed, sessions=sessions, layers=layers, heads=heads, head_dim=64,
                  window=1024, page_rows=16)
    kp, vp, pt, meta = kv.k_pool.to(dev), kv.v_pool.to(dev), kv.page_table.to(dev), kv.meta.to(dev)
    sess = [pcs.kv_session(s, meta[s], kp, vp, pt[s], kv.ring_start[s], kv.window)
            for s in range(sessions)]
    return kv, (kp, vp, pt, meta), sess


def _targets(kv, dev, sessions):
    pt2 = synth.page_permutation(9, sessions, kv.layers, kv.window // kv.page_rows).to(dev)
    k2 = torch.zeros_like(kv.k_pool, device=dev)
    v2 = torch.zeros_like(kv.v_pool, device=dev)
    m2 = torch.zeros_like(kv.meta, device=dev)
    return [pcs.kv_session(s, m2[s], k2, v2, pt2[s], pcs.PCS_RING_START_FROM_SNAPSHOT, kv.window)
            for s in range(sessions)]


def test_many_section_records_equal_the_oracle(ctx, dev):
    kv, _, sess = _kv_setup(dev)
    snaps = ctx.checkpoint(sess)
    assert ctx.info(snaps[0]).n_sections == 2 * kv.layers + 1 > 32
    for s, x in enumerate(snaps):
        ref = oracle.pack(oracle.kv_session(s, kv.meta[s].numpy(), np_view(kv.k_pool),
                                            np_view(kv.v_pool), kv.page_table[s].numpy(),
                                            kv.ring_start[s], kv.window, kv.page_rows,
                                            kv.row_bytes))
        assert np.array_equal(ctx.record(x).numpy(), ref), s
    assert ctx.restore_status(snaps, _targets(kv, dev, len(snaps)), verify=True) == pcs.PCS_OK
    for x in snaps:
        ctx.delete(x)


@pytest.mark.parametrize("where", ["payload", "section_fp", "session_fp"])
def test_many_section_restore_reports_corruption(ctx, dev, tmp_path, where):
    kv, _, sess = _kv_setup(dev, seed=405)
    snaps = ctx.checkpoint(sess)
    victim = 2
    rec = ctx.record(snaps[victim]).numpy().copy()
    sec = 37  # a section past the first 32
    if where == "payload":
        rec[ctx.section(snaps[victim], sec).offset + 777] ^= 0x08
    elif where == "section_fp":
        rec[64 + 64 * sec + 32] ^= 0x01   # the entry's fp field
    else:
        rec[24 + 3] ^= 0x40               # the header's session fp
    path = str(tmp_path / "bad.pcs")
    rec.tofile(path)
    back = ctx.read_file(path)
    group = snaps[:victim] + [back] + snaps[victim + 1:]
    assert ctx.restore_status(group, _targets(kv, dev, len(group)), verify=True) == \
        pcs.PCS_E_CORRUPT
    # The intact records alone still restore verified.
    good = snaps[:victim] + snaps[victim + 1:]
    assert ctx.restore_status(good, _targets(kv, dev, len(good)), verify=True) == pcs.PCS_OK
    for x in snaps + [back]:
        ctx.delete(x)
