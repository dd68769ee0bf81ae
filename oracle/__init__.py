"""Plain CPU oracle for the PCS hot path (test infrastructure only).

Only the test-suite, ``__graft_entry__.smoke()`` and the CPU-baseline /
reference leg of ``bench.py`` may import this package.  It compiles
``pcs_oracle.c`` with gcc (scalar, ``-O1 -ffp-contract=off``, no vector or
fast-math flags) into ``oracle/_build/libpcs_oracle.so`` and exposes its
functions on numpy arrays.  It shares no code with the CUDA library under
``paper_2607_21686_gb300/``: its own record layout description, its own
section structure, its own builders of the three session kinds.

Session kinds (the three PCS shapes of Table tab:pcs, Sec. 7.2):
  markov  {OBS uint8 observation, RNG 16-byte generator state}
  bank    {KEPT_IDX int32[k], KEYS [k][D], VALUES [k][V]}  (kept entries only)
  kv      {META position indices, then K and V of every layer, each the
           window's rows in logical (oldest-first) order}
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pcs_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libpcs_oracle.so")
_lock = threading.Lock()
_lib = None

# Section layouts (how a section's logical rows map to memory).
CONTIG, ROWS, RING = 0, 1, 2
# Element types recorded in section entries (same codes as dtype tags).
DT_RAW, DT_U8, DT_I32, DT_I64, DT_F16, DT_BF16, DT_F32, DT_U64 = 0, 1, 2, 3, 4, 5, 6, 7
# Section types.
SEC_OBS, SEC_RNG, SEC_KEPT_IDX, SEC_KEYS, SEC_VALUES, SEC_META, SEC_K, SEC_V = 1, 2, 3, 4, 5, 6, 7, 8
# Session kinds.
KIND_MARKOV, KIND_BANK, KIND_KV = 1, 2, 3

RING_START_FROM_RECORD = 0xFFFFFFFF
E_CORRUPT = -6


def build(force: bool = False) -> str:
    """Compile the oracle shared library with gcc; return its path."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + ".%d.tmp" % os.getpid()
    cmd = ["gcc", "-std=gnu11", "-O1", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-Wall", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class Section(ctypes.Structure):
    """Mirror of pcso_section in pcs_oracle.c."""
    _fields_ = [
        ("type", ctypes.c_uint32), ("dtype", ctypes.c_uint32),
        ("layer", ctypes.c_uint32), ("layout", ctypes.c_uint32),
        ("base", ctypes.c_void_p), ("bytes", ctypes.c_uint64),
        ("row_bytes", ctypes.c_uint64), ("index", ctypes.c_void_p),
        ("ring_start", ctypes.c_uint32), ("window", ctypes.c_uint32),
        ("page_rows", ctypes.c_uint32), ("reserved", ctypes.c_uint32),
        ("dim0", ctypes.c_uint64), ("dim1", ctypes.c_uint64),
    ]


def lib():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        L = ctypes.CDLL(build())
        u64, u32, i32, vp = ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int32, ctypes.c_void_p
        sig = {
            "pcso_fmix": (u64, [u64]),
            "pcso_comb": (u64, [u64, u64]),
            "pcso_tree": (u64, [vp, u64]),
            "pcso_lane_value": (u64, [vp, u64, u64, ctypes.c_uint]),
            "pcso_chunk_hash": (u64, [vp, u64, u64]),
            "pcso_n_chunks": (u64, [u64]),
            "pcso_fingerprint": (u64, [vp, u64]),
            "pcso_fingerprint_many": (None, [vp, vp, i32, vp]),
            "pcso_classify": (None, [vp, vp, i32, vp]),
            "pcso_score_f32": (ctypes.c_float, [vp, vp, i32, i32]),
            "pcso_score_f64": (ctypes.c_double, [vp, vp, i32, i32]),
            "pcso_score_many": (None, [vp, vp, i32, i32, i32, vp, vp]),
            "pcso_ord32": (u32, [ctypes.c_float]),
            "pcso_key64": (u64, [ctypes.c_float, u32]),
            "pcso_topk": (i32, [vp, i32, i32, vp]),
            "pcso_k_fixed": (None, [vp, i32, i32, vp]),
            "pcso_k_budget": (None, [vp, vp, i32, u64, vp]),
            "pcso_k_fraction": (None, [vp, i32, ctypes.c_double, vp]),
            "pcso_payload_start": (u64, [i32]),
            "pcso_record_bytes": (u64, [vp, i32]),
            "pcso_pack": (u64, [vp, i32, u32, u32, vp, u64]),
            "pcso_record_header": (i32, [vp, vp, vp, vp, vp, vp]),
            "pcso_record_section": (None, [vp, i32, vp, vp, vp, vp]),
            "pcso_restore": (i32, [vp, vp, i32, i32]),
            "pcso_budget_plan": (i32, [vp, vp, vp, i32, u64, ctypes.c_double, vp, vp, vp]),
            "pcso_prune_global": (ctypes.c_int64, [vp, vp, vp, i32, u64, vp, vp]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
        return L


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _bytes_view(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    return a.view(np.uint8).reshape(-1)


# --------------------------------------------------------------------------
# Fingerprint and classification
# --------------------------------------------------------------------------

def fmix(z: int) -> int:
    return lib().pcso_fmix(z & (2**64 - 1))


def comb(a: int, b: int) -> int:
    return lib().pcso_comb(a & (2**64 - 1), b & (2**64 - 1))


def tree(items) -> int:
    v = np.ascontiguousarray(np.asarray(items, dtype=np.uint64))
    assert v.size >= 1
    return lib().pcso_tree(_ptr(v), v.size)


def n_chunks(L: int) -> int:
    return lib().pcso_n_chunks(L)


def lane_value(data, c: int, lane: int, L: int | None = None) -> int:
    b = _bytes_view(data)
    return lib().pcso_lane_value(_ptr(b), b.size if L is None else L, c, lane)


def chunk_hash(data, c: int, L: int | None = None) -> int:
    b = _bytes_view(data)
    return lib().pcso_chunk_hash(_ptr(b), b.size if L is None else L, c)


def fingerprint(data) -> int:
    """PCSFP64-v1 of the bytes of ``data`` (any contiguous numpy array)."""
    b = _bytes_view(data)
    return lib().pcso_fingerprint(_ptr(b) if b.size else 0, b.size)


def fingerprint_many(buffers) -> np.ndarray:
    views = [_bytes_view(x) for x in buffers]
    ptrs = np.array([_ptr(v) if v.size else 0 for v in views], dtype=np.uint64)
    lens = np.array([v.size for v in views], dtype=np.uint64)
    out = np.zeros(len(views), dtype=np.uint64)
    lib().pcso_fingerprint_many(_ptr(ptrs), _ptr(lens), len(views), _ptr(out))
    return out


def classify(fp_before, fp_after) -> np.ndarray:
    a = np.ascontiguousarray(fp_before, dtype=np.uint64)
    b = np.ascontiguousarray(fp_after, dtype=np.uint64)
    out = np.zeros(a.size, dtype=np.uint8)
    lib().pcso_classify(_ptr(a), _ptr(b), a.size, _ptr(out))
    return out


# --------------------------------------------------------------------------
# Relevance score, ranking, k-rules
# --------------------------------------------------------------------------

def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float16:
        return DT_F16
    if a.dtype == np.uint16:  # bfloat16 carried as raw uint16 bits
        return DT_BF16
    raise TypeError("keys/query must be float16, or uint16 holding bfloat16 bits")


def scores(query: np.ndarray, keys: np.ndarray, want64: bool = False):
    """Fixed-order fp32 cosine of each key row against the query (and fp64)."""
    q = np.ascontiguousarray(query)
    k = np.ascontiguousarray(keys)
    dt = _dtype_code(k)
    assert _dtype_code(q) == dt and k.ndim == 2 and q.size == k.shape[1]
    n, D = k.shape
    out32 = np.zeros(n, dtype=np.float32)
    out64 = np.zeros(n, dtype=np.float64) if want64 else None
    lib().pcso_score_many(_ptr(q), _ptr(k), n, D, dt, _ptr(out32),
                          _ptr(out64) if want64 else None)
    return (out32, out64) if want64 else out32


def ord32(s: float) -> int:
    return lib().pcso_ord32(s)


def key64(s: float, idx: int) -> int:
    return lib().pcso_key64(s, idx)


def topk(scores32: np.ndarray, k: int) -> np.ndarray:
    s = np.ascontiguousarray(scores32, dtype=np.float32)
    out = np.zeros(max(min(k, s.size), 0), dtype=np.int32)
    m = lib().pcso_topk(_ptr(s), s.size, k, _ptr(out) if out.size else None)
    assert m == out.size
    return out


def k_fixed(n, k_max: int) -> np.ndarray:
    a = np.ascontiguousarray(n, dtype=np.int32)
    out = np.zeros_like(a)
    lib().pcso_k_fixed(_ptr(a), a.size, k_max, _ptr(out))
    return out


def k_budget(n, entry_bytes, budget: int) -> np.ndarray:
    a = np.ascontiguousarray(n, dtype=np.int32)
    e = np.ascontiguousarray(np.broadcast_to(np.asarray(entry_bytes, dtype=np.uint64), a.shape))
    out = np.zeros_like(a)
    lib().pcso_k_budget(_ptr(a), _ptr(e), a.size, budget, _ptr(out))
    return out


def k_fraction(n, frac: float) -> np.ndarray:
    a = np.ascontiguousarray(n, dtype=np.int32)
    out = np.zeros_like(a)
    lib().pcso_k_fraction(_ptr(a), a.size, frac, _ptr(out))
    return out


def budget_plan(n, entry_bytes, budget: int, frac: float, priority=None):
    """Reactive shrink-then-drop plan: (k per bank, shrinks, drops)."""
    a = np.ascontiguousarray(n, dtype=np.int32)
    e = np.ascontiguousarray(np.broadcast_to(np.asarray(entry_bytes, dtype=np.uint64), a.shape))
    pr = None if priority is None else np.ascontiguousarray(priority, dtype=np.float64)
    k = np.zeros_like(a)
    sh, dr = ctypes.c_int32(), ctypes.c_int32()
    rc = lib().pcso_budget_plan(_ptr(a), _ptr(e), None if pr is None else _ptr(pr), a.size,
                                budget, frac, _ptr(k), ctypes.byref(sh), ctypes.byref(dr))
    assert rc == 0
    return k, sh.value, dr.value


def prune_global(scores32, n, entry_bytes, budget: int):
    """One relevance threshold across all banks under a byte budget.

    Returns (kept indices per bank concatenated, offsets int32[len(n)+1]).
    """
    a = np.ascontiguousarray(n, dtype=np.int32)
    e = np.ascontiguousarray(np.broadcast_to(np.asarray(entry_bytes, dtype=np.uint64), a.shape))
    s = np.ascontiguousarray(scores32, dtype=np.float32)
    assert s.size == int(a.astype(np.int64).sum())
    kept = np.zeros(max(s.size, 1), dtype=np.int32)
    off = np.zeros(a.size + 1, dtype=np.int32)
    m = lib().pcso_prune_global(_ptr(s), _ptr(a), _ptr(e), a.size, budget, _ptr(kept), _ptr(off))
    assert m >= 0 and m == off[-1]
    return kept[:m].copy(), off


# --------------------------------------------------------------------------
# Snapshot records: pack (checkpoint) and restore
# --------------------------------------------------------------------------

class SessionSpec:
    """A session as a list of sections; keeps the numpy arrays alive."""

    def __init__(self, session_id: int, kind: int):
        self.session_id = session_id
        self.kind = kind
        self.sections: list[Section] = []
        self._keep: list = []

    def _add(self, sec: Section, *arrays):
        self.sections.append(sec)
        self._keep.extend(arrays)
        return self

    def contig(self, type_, dtype, arr: np.ndarray, layer=0, dim0=0, dim1=0):
        assert arr.flags.c_contiguous
        s = Section(type=type_, dtype=dtype, layer=layer, layout=CONTIG,
                    base=_ptr(arr) if arr.nbytes else None, bytes=arr.nbytes,
                    dim0=dim0, dim1=dim1)
        return self._add(s, arr)

    def rows(self, type_, dtype, base: np.ndarray, row_bytes: int, index: np.ndarray,
             layer=0, dim0=0, dim1=0):
        assert base.flags.c_contiguous and index.dtype == np.int32
        s = Section(type=type_, dtype=dtype, layer=layer, layout=ROWS,
                    base=_ptr(base), bytes=row_bytes * index.size, row_bytes=row_bytes,
                    index=_ptr(index) if index.size else None, dim0=dim0, dim1=dim1)
        return self._add(s, base, index)

    def ring(self, type_, dtype, pool: np.ndarray, row_bytes: int, page_table: np.ndarray,
             ring_start: int, window: int, page_rows: int, layer=0, dim0=0, dim1=0):
        assert pool.flags.c_contiguous and page_table.dtype == np.int32
        assert window % page_rows == 0 and page_table.size == window // page_rows
        s = Section(type=type_, dtype=dtype, layer=layer, layout=RING,
                    base=_ptr(pool), bytes=row_bytes * window, row_bytes=row_bytes,
                    index=_ptr(page_table), ring_start=ring_start & 0xFFFFFFFF,
                    window=window, page_rows=page_rows, dim0=dim0, dim1=dim1)
        return self._add(s, pool, page_table)

    def array(self):
        arr = (Section * len(self.sections))(*self.sections)
        return arr


def record_bytes(spec: SessionSpec) -> int:
    arr = spec.array()
    return lib().pcso_record_bytes(ctypes.addressof(arr), len(spec.sections))


def payload_start(n_sections: int) -> int:
    return lib().pcso_payload_start(n_sections)


def pack(spec: SessionSpec) -> np.ndarray:
    """checkpoint(s): the PCS1 record of one session as a uint8 array."""
    arr = spec.array()
    n = len(spec.sections)
    total = lib().pcso_record_bytes(ctypes.addressof(arr), n)
    out = np.empty(total, dtype=np.uint8)
    got = lib().pcso_pack(ctypes.addressof(arr), n, spec.session_id, spec.kind, _ptr(out), total)
    assert got == total, (got, total)
    return out


def restore(record: np.ndarray, targets: SessionSpec, verify: bool = True) -> int:
    """restore(c) into the target sections; returns 0, -1 (shape) or -6 (corrupt)."""
    rec = np.ascontiguousarray(record, dtype=np.uint8)
    arr = targets.array()
    return lib().pcso_restore(_ptr(rec), ctypes.addressof(arr), len(targets.sections),
                              1 if verify else 0)


def record_header(record: np.ndarray) -> dict:
    rec = np.ascontiguousarray(record, dtype=np.uint8)
    ns, sid, kind = ctypes.c_uint32(), ctypes.c_uint32(), ctypes.c_uint32()
    total, sfp = ctypes.c_uint64(), ctypes.c_uint64()
    ok = lib().pcso_record_header(_ptr(rec), ctypes.byref(ns), ctypes.byref(sid),
                                  ctypes.byref(kind), ctypes.byref(total), ctypes.byref(sfp))
    if not ok:
        raise ValueError("not a PCS1 record")
    return dict(n_sections=ns.value, session_id=sid.value, kind=kind.value,
                total_bytes=total.value, session_fp=sfp.value)


def record_section(record: np.ndarray, i: int) -> dict:
    rec = np.ascontiguousarray(record, dtype=np.uint8)
    off, nb, fp, aux = (ctypes.c_uint64() for _ in range(4))
    lib().pcso_record_section(_ptr(rec), i, ctypes.byref(off), ctypes.byref(nb),
                              ctypes.byref(fp), ctypes.byref(aux))
    return dict(offset=off.value, bytes=nb.value, fp=fp.value, aux=aux.value)


# --------------------------------------------------------------------------
# Builders of the three session kinds (Table tab:pcs shapes)
# --------------------------------------------------------------------------

def markov_session(session_id: int, obs: np.ndarray, rng_state: np.ndarray) -> SessionSpec:
    """{observation uint8, generator state: seed u64 then offset u64}."""
    assert obs.dtype == np.uint8 and rng_state.dtype == np.uint64 and rng_state.size == 2
    sp = SessionSpec(session_id, KIND_MARKOV)
    sp.contig(SEC_OBS, DT_U8, obs, dim0=obs.size)
    sp.contig(SEC_RNG, DT_U64, rng_state, dim0=2)
    return sp


def bank_session(session_id: int, keys: np.ndarray, values: np.ndarray,
                 kept: np.ndarray, key_dtype: int, value_dtype: int) -> SessionSpec:
    """{KEPT_IDX int32[k], KEYS [k][D] gathered, VALUES [k][V] gathered}."""
    kept = np.ascontiguousarray(kept, dtype=np.int32)
    kb = keys.reshape(keys.shape[0], -1).view(np.uint8).shape[1]
    vb = values.reshape(values.shape[0], -1).view(np.uint8).shape[1]
    sp = SessionSpec(session_id, KIND_BANK)
    sp.contig(SEC_KEPT_IDX, DT_I32, kept, dim0=kept.size)
    sp.rows(SEC_KEYS, key_dtype, keys, kb, kept, dim0=kept.size, dim1=kb)
    sp.rows(SEC_VALUES, value_dtype, values, vb, kept, dim0=kept.size, dim1=vb)
    return sp


def bank_targets(session_id: int, kept_out: np.ndarray, keys_out: np.ndarray,
                 values_out: np.ndarray, key_dtype: int, value_dtype: int) -> SessionSpec:
    """Restore targets of a bank record: the compacted bank (kept rows only)."""
    k = kept_out.size
    sp = SessionSpec(session_id, KIND_BANK)
    sp.contig(SEC_KEPT_IDX, DT_I32, kept_out, dim0=k)
    sp.contig(SEC_KEYS, key_dtype, keys_out, dim0=k)
    sp.contig(SEC_VALUES, value_dtype, values_out, dim0=k)
    return sp


def kv_session(session_id: int, meta: np.ndarray, k_pool: np.ndarray, v_pool: np.ndarray,
               page_table: np.ndarray, ring_start: int, window: int, page_rows: int,
               row_bytes: int, ring_start_override: int | None = None,
               v_page_table: np.ndarray | None = None) -> SessionSpec:
    """{META, then K_l, V_l for each layer l}; page_table is int32 [layers][pages]
    (of K, and of V unless v_page_table is given)."""
    layers = page_table.shape[0]
    vt = page_table if v_page_table is None else v_page_table
    sp = SessionSpec(session_id, KIND_KV)
    sp.contig(SEC_META, DT_I64, meta, dim0=meta.size)
    rs = ring_start if ring_start_override is None else ring_start_override
    for l in range(layers):
        pt = np.ascontiguousarray(page_table[l], dtype=np.int32)
        pv = np.ascontiguousarray(vt[l], dtype=np.int32)
        sp.ring(SEC_K, DT_BF16, k_pool, row_bytes, pt, rs, window, page_rows, layer=l,
                dim0=window, dim1=row_bytes)
        sp.ring(SEC_V, DT_BF16, v_pool, row_bytes, pv, rs, window, page_rows, layer=l,
                dim0=window, dim1=row_bytes)
    return sp


# --------------------------------------------------------------------------
# Copy-on-write page pool (Sec. 3, I3: the mechanism realises fork
# independence by copy-on-write; Sec. 3 "Boundary": the runtime owns
# allocation and copy-on-write; Sec. 7.3: ref-counted blocks whose copy leg
# fires on the first write).  Sequential reference model.
# --------------------------------------------------------------------------

class PoolError(Exception):
    pass


class PagePool:
    """n_pages pages of page_bytes; a reference count per page; free stack.

    alloc(n)               -> n fresh pages, count 1 each (lowest ids first)
    share(ids)             -> the same ids, every valid page count + 1 (a fork
                              of the tables that hold them: no bytes move)
    prepare_write(t, e)    -> before writing table entries t[e]: an entry whose
                              page is held elsewhere (count > 1) gets a fresh
                              copy of it and gives up its hold; a page held by
                              this entry alone is kept as it is
    release(ids)           -> every valid page count - 1; pages at 0 are free
    Page id -1 marks an empty table slot and is skipped everywhere.
    """

    def __init__(self, n_pages: int, page_bytes: int):
        self.data = np.zeros((n_pages, page_bytes), dtype=np.uint8)
        self.rc = np.zeros(n_pages, dtype=np.int64)
        self.free = list(range(n_pages - 1, -1, -1))  # pop() gives the lowest id
        self.copies = 0

    def _pop(self) -> int:
        if not self.free:
            raise PoolError("no free page")
        q = self.free.pop()
        self.rc[q] = 1
        return q

    def alloc(self, n: int) -> np.ndarray:
        return np.array([self._pop() for _ in range(n)], dtype=np.int32)

    def share(self, ids) -> np.ndarray:
        ids = np.asarray(ids, dtype=np.int32)
        for p in ids.reshape(-1).tolist():
            if p >= 0:
                self.rc[p] += 1
        return ids.copy()

    def prepare_write(self, table: np.ndarray, entries=None) -> None:
        flat = table.reshape(-1)
        todo = range(flat.size) if entries is None else np.asarray(entries).reshape(-1).tolist()
        for e in todo:
            p = int(flat[e])
            if p < 0 or self.rc[p] == 1:
                continue
            q = self._pop()
            self.data[q] = self.data[p]
            self.rc[p] -= 1
            flat[e] = q
            self.copies += 1

    def release(self, ids) -> None:
        for p in np.asarray(ids).reshape(-1).tolist():
            if p < 0:
                continue
            if self.rc[p] <= 0:
                raise PoolError("page %d released more often than held" % p)
            self.rc[p] -= 1
            if self.rc[p] == 0:
                self.free.append(p)

    def gather(self, table) -> np.ndarray:
        """The bytes a table addresses, in table order (empty slots skipped)."""
        ids = [p for p in np.asarray(table).reshape(-1).tolist() if p >= 0]
        return self.data[ids].reshape(-1).copy()


# --------------------------------------------------------------------------
# State versus witness (Sec. 3, "A distinction the implementation forced"):
# a buffer is PCS iff restore reads it.  Given the byte ranges a restore
# read, a buffer is "read" iff some read of at least one byte overlaps it.
# --------------------------------------------------------------------------

def classify_reads(bufs, reads) -> np.ndarray:
    """bufs, reads: sequences of (address, bytes); returns uint8 flags per buffer."""
    flags = np.zeros(len(bufs), dtype=np.uint8)
    for i, (b, nb) in enumerate(bufs):
        for r, nr in reads:
            if nb > 0 and nr > 0 and r < b + nb and b < r + nr:
                flags[i] = 1
                break
    return flags


# --------------------------------------------------------------------------
# Discovering PCS by measurement (Sec. 4, procedure FINGERPRINT):
#   1. necessity: for each component, snapshot all the others, run the probe,
#      measure D; the component is necessary if D > eps;
#   2. sufficiency: snapshot exactly the necessary set N; if D <= eps, PCS = N;
#   3. redundancy fallback: otherwise greedily add the component that most
#      reduces D until D <= eps;
#   4. PCS and Derivable = the rest.
# D here is a count of differing output bytes (eps = 0: byte identity).
# --------------------------------------------------------------------------

def mismatch(a, b) -> int:
    """Bytes that differ between a and b, counting every byte past the shorter."""
    a, b = _bytes_view(a), _bytes_view(b)
    m = min(a.size, b.size)
    return int(np.count_nonzero(a[:m] != b[:m])) + abs(a.size - b.size)


def discover(k: int, probe, eps: int):
    """probe(keep: list[bool]) -> D.  Returns (pcs flags, probes run, consistent)."""
    probes = 0

    def run(keep):
        nonlocal probes
        probes += 1
        return probe(list(keep))

    necessary = []
    for i in range(k):
        keep = [j != i for j in range(k)]
        necessary.append(run(keep) > eps)
    chosen = list(necessary)
    d = run(chosen)
    while d > eps and not all(chosen):
        best_j, best_d = -1, None
        for j in range(k):
            if chosen[j]:
                continue
            dj = run([c or (x == j) for x, c in enumerate(chosen)])
            if best_d is None or dj < best_d:
                best_j, best_d = j, dj
        chosen[best_j] = True
        d = best_d
    return np.array(chosen, dtype=np.uint8), probes, d <= eps
