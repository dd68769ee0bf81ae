"""Second, structurally different statements of the oracle's lane chain and
fixed-order fp32 score, and the slips they catch (CPU only).

The fingerprint PCSFP64-v1 and the score's summation order are frozen
readings (the paper prints neither a hash nor a relevance formula; Sec. 4
step 1 needs a content fingerprint, Sec. 5 / Sec. 7.5 a relevance rank).  The
oracle states them as scalar C loops over (lane, segment, word) and
(element, lane).  Here they are stated again from the definition alone, in
another shape, with no oracle code on the path:

* the chain runs on all 32 lanes at once: a 4 KiB chunk viewed as
  u64[8][32][2] is [k][lane][word of the segment] -- segment s = lane + 32k
  holds words 2s and 2s+1, i.e. word 64k + 2*lane + j -- and every step is a
  numpy uint64 vector operation (wrapping multiply, shift-or rotate);
* the buffer tree is the top-down split (left part = the largest power of two
  below the length), not the bottom-up levels of the oracle;
* the score views a padded key as float32[blocks][32 lanes][8] (element
  e = 256*block + 8*lane + i, so lane = floor(e/8) mod 32) and accumulates
  lane vectors block by block, element by element, in numpy float32 (each
  product and each sum rounded to binary32, as the definition orders).

Each is compared with the oracle bit for bit, and then the slips a reader
could make in the oracle (a rotation of 31 for 23, the two words of a segment
swapped, another seed, contiguous segments per lane, a lane map of e mod 32,
a sequential sum, the lane tree folded in halves) are planted in a
copy of the oracle compiled on the CPU: each must fail a comparison here.
"""
import ctypes
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle

M64 = (1 << 64) - 1
P = np.uint64(0x9E3779B97F4A7C15)
SEED = np.uint64(0x5043534650363401)
FMIX_M1 = np.uint64(0xBF58476D1CE4E5B9)
FMIX_M2 = np.uint64(0x94D049BB133111EB)


# --------------------------------------------------------------------------
# Fingerprint, vectorised over the 32 lanes
# --------------------------------------------------------------------------

def _v_fmix(z):
    z = np.asarray(z, dtype=np.uint64).copy()
    z ^= z >> np.uint64(30)
    z *= FMIX_M1
    z ^= z >> np.uint64(27)
    z *= FMIX_M2
    z ^= z >> np.uint64(31)
    return z


def _v_rotl(x, r):
    return (x << np.uint64(r)) | (x >> np.uint64(64 - r))


def _v_comb(a, b):
    return _v_fmix(np.asarray(a, np.uint64) * P + _v_rotl(np.asarray(b, np.uint64), 31))


def _chunk_words(data: np.ndarray, c: int) -> np.ndarray:
    """Chunk c as u64[8][32][2] (k, lane, j), bytes past the end read as 0."""
    raw = np.zeros(4096, dtype=np.uint8)
    piece = data[4096 * c: 4096 * (c + 1)]
    raw[:piece.size] = piece
    return raw.view("<u8").reshape(8, 32, 2)


def lane_values(data: np.ndarray, c: int) -> np.ndarray:
    """a_l of chunk c for all 32 lanes at once (u64[32])."""
    W = _chunk_words(data, c)
    with np.errstate(over="ignore"):
        h = _v_fmix(SEED ^ (np.uint64(32 * c) + np.arange(32, dtype=np.uint64)))
        for k in range(8):
            for j in range(2):
                h = (_v_rotl(h, 23) ^ W[k, :, j]) * P
        return _v_fmix(h)


def chunk_hash(data: np.ndarray, c: int) -> int:
    v = lane_values(data, c)
    with np.errstate(over="ignore"):
        d = 1
        while d < 32:
            v[0::2 * d] = _v_comb(v[0::2 * d], v[d::2 * d])
            d *= 2
    return int(v[0])


def _tree_split(xs):
    if len(xs) == 1:
        return xs[0]
    h = 1
    while 2 * h < len(xs):
        h *= 2
    with np.errstate(over="ignore"):
        return int(_v_comb(np.uint64(_tree_split(xs[:h])), np.uint64(_tree_split(xs[h:]))))


def fingerprint(data: np.ndarray) -> int:
    L = data.size
    C = max(1, -(-L // 4096))
    root = _tree_split([chunk_hash(data, c) for c in range(C)])
    with np.errstate(over="ignore"):
        return int(_v_fmix(np.uint64(root) ^ np.uint64((L * int(P)) & M64)))


# --------------------------------------------------------------------------
# Score, vectorised over the 32 lanes
# --------------------------------------------------------------------------

def _as_f32(bits: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "f16":
        return bits.view(np.float16).astype(np.float32)          # exact
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)  # exact


def score(q_bits: np.ndarray, k_bits: np.ndarray, dtype: str) -> np.float32:
    D = q_bits.size
    blocks = -(-D // 256)
    qv = np.zeros(256 * blocks, np.float32)
    kv = np.zeros(256 * blocks, np.float32)
    qv[:D] = _as_f32(q_bits, dtype)
    kv[:D] = _as_f32(k_bits, dtype)
    qv = qv.reshape(blocks, 32, 8)
    kv = kv.reshape(blocks, 32, 8)
    sd = np.zeros(32, np.float32)
    sq = np.zeros(32, np.float32)
    sk = np.zeros(32, np.float32)
    # Padding elements add +0 products to sums that start at +0: no change.
    for b in range(blocks):
        for i in range(8):
            qe, ke = qv[b, :, i], kv[b, :, i]
            sd = sd + qe * ke
            sq = sq + qe * qe
            sk = sk + ke * ke
    d = 1
    while d < 32:
        sd[0::2 * d] = sd[0::2 * d] + sd[d::2 * d]
        sq[0::2 * d] = sq[0::2 * d] + sq[d::2 * d]
        sk[0::2 * d] = sk[0::2 * d] + sk[d::2 * d]
        d *= 2
    den = np.sqrt(sq[0]) * np.sqrt(sk[0])   # float32 sqrt and product, RN
    if den == np.float32(0):
        return np.float32(0)
    return np.float32(sd[0] / den)


# --------------------------------------------------------------------------
# The restatements agree with the oracle
# --------------------------------------------------------------------------

def _rand_bytes(seed, n):
    return np.random.default_rng(seed).integers(0, 256, n, dtype=np.uint8)


def test_restated_fmix_is_splitmix64():
    # The vector mixer against the published SplitMix64 stream for state 0.
    with open(os.path.join(os.path.dirname(__file__), "golden", "splitmix64_seed0.txt")) as f:
        expected = [int(t.split()[0], 16) for t in f if t.strip() and not t.startswith("#")]
    states = (np.arange(1, len(expected) + 1, dtype=np.uint64) * P)
    with np.errstate(over="ignore"):
        assert [int(x) for x in _v_fmix(states)] == expected


@pytest.mark.parametrize("c", [0, 1, 5, 1000])
def test_lane_chain_matches_oracle(c):
    data = _rand_bytes(100 + c, 4096 * (c + 1))
    mine = lane_values(data, c)
    theirs = [oracle.lane_value(data, c, l) for l in range(32)]
    assert [int(x) for x in mine] == theirs


def test_lane_chain_zero_padded_tail():
    # A chunk that ends mid-segment: the missing bytes read as zero.
    data = _rand_bytes(7, 4096 + 1234)
    mine = lane_values(data, 1)
    assert [int(x) for x in mine] == [oracle.lane_value(data, 1, l) for l in range(32)]
    assert chunk_hash(data, 1) == oracle.chunk_hash(data, 1)


@pytest.mark.parametrize("L", [0, 1, 8, 15, 16, 4095, 4096, 4097, 3 * 4096 + 5, 9 * 4096 + 777])
def test_fingerprint_matches_oracle(L):
    data = _rand_bytes(L + 31, L)
    assert fingerprint(data) == oracle.fingerprint(data)


def _score_inputs(seed, n, D, dtype):
    rnd = np.random.default_rng(seed)
    if dtype == "f16":
        q = rnd.standard_normal(D).astype(np.float16).view(np.uint16)
        k = rnd.standard_normal((n, D)).astype(np.float16).view(np.uint16)
    else:  # bf16 bit patterns: round-to-nearest-even of float32 samples
        def bf(a):
            u = a.astype(np.float32).view(np.uint32).astype(np.uint64)
            u = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
            return u.astype(np.uint16)
        q = bf(rnd.standard_normal(D))
        k = bf(rnd.standard_normal((n, D)))
    return q, k


def _oracle_scores(q, k, dtype):
    if dtype == "f16":
        return oracle.scores(q.view(np.float16), k.view(np.float16))
    return oracle.scores(q, k)


@pytest.mark.parametrize("dtype,D", [("f16", 256), ("bf16", 512), ("f16", 8), ("bf16", 40),
                                     ("f16", 264), ("bf16", 1000)])
def test_score_order_matches_oracle_bit_for_bit(dtype, D):
    q, k = _score_inputs(D * 7 + len(dtype), 64, D, dtype)
    mine = np.array([score(q, k[i], dtype) for i in range(k.shape[0])], np.float32)
    theirs = _oracle_scores(q, k, dtype)
    assert np.array_equal(mine.view(np.uint32), theirs.view(np.uint32))


def test_score_zero_key_and_extremes():
    q, k = _score_inputs(3, 4, 256, "f16")
    k[0] = 0
    k[1] = np.float16(65504).view(np.uint16)   # largest finite half
    k[2] = np.float16(2 ** -24).view(np.uint16)  # smallest subnormal half
    mine = np.array([score(q, k[i], "f16") for i in range(4)], np.float32)
    theirs = _oracle_scores(q, k, "f16")
    assert np.array_equal(mine.view(np.uint32), theirs.view(np.uint32))
    assert mine[0] == 0


# --------------------------------------------------------------------------
# Planted slips: a copy of the oracle with one plausible mistake must fail
# --------------------------------------------------------------------------

_SRC = os.path.join(os.path.dirname(oracle.__file__), "pcs_oracle.c")

# (name, text in the oracle, replacement): each is a reading error a reader
# of the definition could make.
_SLIPS = [
    ("rotation 31 for 23", "rotl64(h, 23)", "rotl64(h, 31)"),
    ("words of a segment swapped", "16u * seg + 8u * j", "16u * seg + 8u * (1u - j)"),
    ("seed off by one bit", "0x5043534650363401ull", "0x5043534650363400ull"),
    ("segments contiguous per lane", "uint64_t seg = lane + PCSO_LANES * k;",
     "uint64_t seg = PCSO_SEGS_PER_LANE * lane + k;"),
    ("lane index without the chunk", "PCSO_SEED ^ (c * PCSO_LANES + lane)", "PCSO_SEED ^ lane"),
    ("score lane map e mod 32", "l = (unsigned)((e / 8) % PCSO_LANES);",
     "l = (unsigned)(e % PCSO_LANES);"),
    ("score summed sequentially", "l = (unsigned)((e / 8) % PCSO_LANES);", "l = 0;"),
    ("score lane tree folded in halves",
     "for (d = 1; d < PCSO_LANES; d *= 2)\n        for (l = 0; l < PCSO_LANES; l += 2 * d) {",
     "for (d = PCSO_LANES / 2; d >= 1; d /= 2)\n        for (l = 0; l < d; l++) {"),
]


def _build_mutant(tmp_path, name, old, new):
    src = open(_SRC).read()
    assert src.count(old) == 1, name
    path = tmp_path / ("mut_%d.c" % abs(hash(name)))
    path.write_text(src.replace(old, new))
    so = tmp_path / (path.stem + ".so")
    subprocess.run(["gcc", "-std=gnu11", "-O1", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
                    "-shared", "-o", str(so), str(path), "-lm"], check=True)
    L = ctypes.CDLL(str(so))
    L.pcso_fingerprint.restype = ctypes.c_uint64
    L.pcso_fingerprint.argtypes = [ctypes.c_void_p, ctypes.c_uint64]
    L.pcso_score_f32.restype = ctypes.c_float
    L.pcso_score_f32.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32]
    return L


def _agrees(L) -> bool:
    """Whether a compiled oracle variant agrees with the restatements."""
    for n in (4096, 3 * 4096 + 5):
        data = _rand_bytes(n, n)
        if L.pcso_fingerprint(data.ctypes.data, data.size) != fingerprint(data):
            return False
    for dtype, code, D in (("f16", oracle.DT_F16, 256), ("bf16", oracle.DT_BF16, 512)):
        q, k = _score_inputs(D, 16, D, dtype)
        for i in range(k.shape[0]):
            row = np.ascontiguousarray(k[i])
            got = np.float32(L.pcso_score_f32(q.ctypes.data, row.ctypes.data, D, code))
            if got.view(np.uint32) != score(q, row, dtype).view(np.uint32):
                return False
    return True


@pytest.mark.skipif(shutil.which("gcc") is None, reason="gcc needed to build oracle variants")
def test_unmodified_copy_agrees(tmp_path):
    assert _agrees(_build_mutant(tmp_path, "none", "PCSO_CHUNK_BYTES 4096u",
                                 "PCSO_CHUNK_BYTES 4096u"))


@pytest.mark.skipif(shutil.which("gcc") is None, reason="gcc needed to build oracle variants")
@pytest.mark.parametrize("slip", _SLIPS, ids=[s[0] for s in _SLIPS])
def test_planted_slip_is_caught(tmp_path, slip):
    assert not _agrees(_build_mutant(tmp_path, *slip))
