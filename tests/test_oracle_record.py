"""Pins of the oracle's checkpoint (pack) and restore (CPU only).

Pinned to what the paper fixes: the invariants of the contract (Sec. 3) --
I1 round-trip after an excursion that overwrites every source byte, I2 a
checkpoint is an immutable snapshot, I3 fork independence, I4 the snapshot
holds exactly the selected sections -- and the byte counts of Table tab:pcs.
Expected bytes are rebuilt independently here with numpy gathers.
"""
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _np(t):
    t = t.contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def _u8(a):
    return np.ascontiguousarray(a).view(np.uint8).reshape(-1)


def _parse(rec):
    h = oracle.record_header(rec)
    secs = [oracle.record_section(rec, i) for i in range(h["n_sections"])]
    return h, secs


def _check_layout(rec, payloads):
    """I4: exactly these payloads, 256-aligned, zero padding, correct fps."""
    h, secs = _parse(rec)
    assert h["total_bytes"] == rec.size
    assert len(secs) == len(payloads)
    start = oracle.payload_start(len(payloads))
    assert start == -(-(64 + 64 * len(payloads)) // 256) * 256
    covered = np.zeros(rec.size, dtype=bool)
    covered[:64 + 64 * len(payloads)] = True
    off = start
    for s, p in zip(secs, payloads):
        assert s["offset"] == off and s["offset"] % 256 == 0
        assert s["bytes"] == p.size
        assert np.array_equal(rec[off:off + p.size], p)
        assert s["fp"] == oracle.fingerprint(p)
        covered[off:off + p.size] = True
        off = -(-(off + p.size) // 256) * 256
    assert off == rec.size
    assert not rec[~covered].any(), "padding bytes must be zero"
    fps = [s["fp"] for s in secs]
    assert h["session_fp"] == oracle.fmix(oracle.tree(fps) ^ len(fps))


def test_markov_round_trip_after_excursion():
    m = synth.markov(seed=1)
    obs, rng = _np(m.obs), _np(m.rng).view(np.uint64)
    want_obs, want_rng = obs.copy(), rng.copy()
    rec = oracle.pack(oracle.markov_session(7, obs, rng))
    _check_layout(rec, [_u8(want_obs), _u8(want_rng)])
    h = oracle.record_header(rec)
    assert (h["session_id"], h["kind"]) == (7, oracle.KIND_MARKOV)
    # Excursion overwrites every source byte (I2: the snapshot is unaffected).
    rec_before = rec.copy()
    synth.excursion(m, seed=99)
    obs[...] = _np(m.obs)
    rng[...] = _np(m.rng).view(np.uint64)
    assert not np.array_equal(obs, want_obs)
    assert np.array_equal(rec, rec_before)
    assert oracle.restore(rec, oracle.markov_session(7, obs, rng)) == 0
    assert np.array_equal(obs, want_obs) and np.array_equal(rng, want_rng)


def test_markov_rng_bit_flip_changes_fingerprints():
    # Wrong-value control (Sec. 4): corrupting only the RNG must be visible.
    m = synth.markov(seed=2)
    obs, rng = _np(m.obs), _np(m.rng).view(np.uint64).copy()
    rec = oracle.pack(oracle.markov_session(0, obs, rng))
    for bit in [0, 1, 63, 64, 100, 127]:
        r2 = rng.copy()
        r2.view(np.uint8)[bit // 8] ^= np.uint8(1 << (bit % 8))
        assert oracle.fingerprint(r2) != oracle.fingerprint(rng)
        rec2 = oracle.pack(oracle.markov_session(0, obs, r2))
        assert oracle.record_header(rec2)["session_fp"] != oracle.record_header(rec)["session_fp"]


def test_paper_markov_sizes():
    # Table tab:pcs: obs 1,382,400 B (3 x 480 x 960 uint8) + rng 8 B = 1,382,408 B.
    g = {}
    with open(os.path.join(GOLDEN, "pcs_sizes.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, v = line.split()
                g[k] = int(v)
    obs = np.zeros((g["obs_channels"], g["obs_height"], g["obs_width"]), dtype=np.uint8)
    rng8 = np.zeros(1, dtype=np.uint64)
    sp = oracle.SessionSpec(0, oracle.KIND_MARKOV)
    sp.contig(oracle.SEC_OBS, oracle.DT_U8, obs)
    sp.contig(oracle.SEC_RNG, oracle.DT_U64, rng8)
    rec = oracle.pack(sp)
    _, secs = _parse(rec)
    assert secs[0]["bytes"] == g["obs_bytes"]
    assert secs[1]["bytes"] == g["rng_bytes"]
    assert secs[0]["bytes"] + secs[1]["bytes"] == g["pcs_total_bytes"]
    # Record = 256 B of header/table + payloads rounded to 256 B each.
    assert rec.size == 256 + 1382400 + 256


def _bank_case(seed, sessions=5, n_lo=1, n_hi=40, k_max=16):
    b = synth.banks(seed, sessions, n_lo, n_hi, 64, torch.float16, (4, 8), torch.bfloat16)
    return b, oracle.k_fixed(b.n, k_max)


def test_bank_prune_pack_restore():
    b, ks = _bank_case(3)
    keys, vals, qs = _np(b.keys), _np(b.values), _np(b.queries)
    for s in range(b.sessions):
        lo, hi = b.entry_off[s], b.entry_off[s + 1]
        sk = np.ascontiguousarray(keys[lo:hi])
        sv = np.ascontiguousarray(vals[lo:hi])
        sc = oracle.scores(qs[s], sk)
        kept = oracle.topk(sc, int(ks[s]))
        assert kept.size == min(b.n[s], 16) and np.all(np.diff(kept) > 0)
        rec = oracle.pack(oracle.bank_session(s, sk, sv, kept, oracle.DT_F16, oracle.DT_BF16))
        want_k, want_v = sk[kept], sv[kept]
        _check_layout(rec, [_u8(kept), _u8(want_k), _u8(want_v)])
        # Excursion: the live bank is overwritten; restore the compacted bank.
        sk[...] = 0
        sv[...] = 0
        out_i = np.full(kept.size, -1, np.int32)
        out_k = np.zeros_like(want_k)
        out_v = np.zeros_like(want_v)
        t = oracle.bank_targets(s, out_i, out_k, out_v, oracle.DT_F16, oracle.DT_BF16)
        assert oracle.restore(rec, t) == 0
        assert np.array_equal(out_i, kept)
        assert np.array_equal(out_k, want_k) and np.array_equal(out_v, want_v)


def test_bank_with_nothing_kept():
    b, _ = _bank_case(4, sessions=1)
    keys, vals = _np(b.keys), _np(b.values)
    kept = np.zeros(0, np.int32)
    rec = oracle.pack(oracle.bank_session(0, keys, vals, kept, oracle.DT_F16, oracle.DT_BF16))
    _check_layout(rec, [np.zeros(0, np.uint8)] * 3)
    assert rec.size == 256


def _kv_logical(pool, page_table, ring_start, window, page_rows):
    """Independent gather of one ring section in logical order (numpy)."""
    j = np.arange(window)
    slot = (ring_start + j) % window
    page = page_table[slot // page_rows]
    return pool[page, slot % page_rows]


@pytest.mark.parametrize("ring_start", [0, 15, 16, 17, 63])
def test_kv_round_trip_into_fresh_pool(ring_start):
    kv = synth.kv(seed=5, sessions=2, layers=3, heads=2, head_dim=8, window=64, page_rows=16)
    kp, vp = _np(kv.k_pool), _np(kv.v_pool)
    pt = kv.page_table.numpy()
    meta = kv.meta.numpy()
    rb = kv.row_bytes
    for s in range(kv.sessions):
        sp = oracle.kv_session(s, np.ascontiguousarray(meta[s]), kp, vp, pt[s], ring_start,
                               kv.window, kv.page_rows, rb)
        rec = oracle.pack(sp)
        payloads = [_u8(meta[s])]
        for l in range(kv.layers):
            payloads.append(_u8(_kv_logical(kp, pt[s, l], ring_start, kv.window, kv.page_rows)))
            payloads.append(_u8(_kv_logical(vp, pt[s, l], ring_start, kv.window, kv.page_rows)))
        _check_layout(rec, payloads)
        _, secs = _parse(rec)
        assert all(x["aux"] == ring_start for x in secs[1:])
        # Restore into a freshly permuted pool, same ring start (from the record).
        pt2 = synth.page_permutation(77 + s, kv.sessions, kv.layers, kv.window // kv.page_rows)
        pt2 = pt2.numpy()
        kp2, vp2 = np.zeros_like(kp), np.zeros_like(vp)
        meta2 = np.zeros(4, np.int64)
        t = oracle.kv_session(s, meta2, kp2, vp2, pt2[s], 0, kv.window, kv.page_rows, rb,
                              ring_start_override=oracle.RING_START_FROM_RECORD)
        assert oracle.restore(rec, t) == 0
        assert np.array_equal(meta2, meta[s])
        for l in range(kv.layers):
            assert np.array_equal(_kv_logical(kp2, pt2[s, l], ring_start, 64, 16),
                                  _kv_logical(kp, pt[s, l], ring_start, 64, 16))
            assert np.array_equal(_kv_logical(vp2, pt2[s, l], ring_start, 64, 16),
                                  _kv_logical(vp, pt[s, l], ring_start, 64, 16))


def test_verify_detects_corruption_and_shape_mismatch():
    m = synth.markov(seed=6, shape=(3, 16, 16))
    obs, rng = _np(m.obs), _np(m.rng).view(np.uint64)
    rec = oracle.pack(oracle.markov_session(1, obs, rng))
    _, secs = _parse(rec)
    for where in [secs[0]["offset"], secs[0]["offset"] + 700, secs[1]["offset"] + 15]:
        bad = rec.copy()
        bad[where] ^= 1
        assert oracle.restore(bad, oracle.markov_session(1, obs.copy(), rng.copy())) == -6
        # Without verification the corrupt bytes are written back as they are.
        assert oracle.restore(bad, oracle.markov_session(1, obs.copy(), rng.copy()),
                              verify=False) == 0
    bad = rec.copy()
    bad[64 + 32] ^= 1   # a stored section fp
    assert oracle.restore(bad, oracle.markov_session(1, obs.copy(), rng.copy())) == -6
    small = np.zeros(10, np.uint8)
    assert oracle.restore(rec, oracle.markov_session(1, small, rng.copy())) == -1


def test_fork_is_independent():
    # I3: a fork is a byte copy; changing the child leaves the parent intact.
    m = synth.markov(seed=8, shape=(3, 32, 32))
    obs, rng = _np(m.obs), _np(m.rng).view(np.uint64)
    parent = oracle.pack(oracle.markov_session(2, obs, rng))
    child = parent.copy()
    snapshot_of_parent = parent.copy()
    obs2 = obs.copy()
    assert oracle.restore(child, oracle.markov_session(2, obs2, rng.copy())) == 0
    obs2[0, 0, :5] ^= 0xFF
    child[:] = oracle.pack(oracle.markov_session(2, obs2, rng))
    assert np.array_equal(parent, snapshot_of_parent)
    assert oracle.record_header(child)["session_fp"] != oracle.record_header(parent)["session_fp"]
