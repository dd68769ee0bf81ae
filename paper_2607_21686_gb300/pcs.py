"""ctypes binding of libpcs (include/pcs.h): argument marshalling only.

Every step of the path runs in the library's sm_103a kernels; this module
turns torch tensors into pointers, sizes and streams and checks status
codes.  There is no fallback: if ``libpcs.so`` has not been built, importing
the library raises.

The low-level functions keep the C names (``pcs_fingerprint``,
``pcs_checkpoint``, ...).  ``Context`` wraps them for tensors, and the
``*_session`` helpers describe the three session kinds of Table tab:pcs
(Sec. 7.2) as section lists:
  markov  {OBS uint8 observation, RNG 16-byte generator state}
  bank    {KEPT_IDX int32[k], KEYS [k][D], VALUES [k][V]}
  kv      {META position indices, K_l and V_l of every layer in logical order}
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libpcs.so")

PCS_OK = 0
PCS_E_INVAL, PCS_E_ALIGN, PCS_E_NOMEM, PCS_E_CUDA, PCS_E_BUDGET = -1, -2, -3, -4, -5
PCS_E_CORRUPT, PCS_E_HANDLE, PCS_E_IO, PCS_E_TIMEOUT, PCS_E_RANGE = -6, -7, -8, -9, -10

PCS_DT_RAW, PCS_DT_U8, PCS_DT_I32, PCS_DT_I64 = 0, 1, 2, 3
PCS_DT_F16, PCS_DT_BF16, PCS_DT_F32, PCS_DT_U64 = 4, 5, 6, 7
PCS_SEC_OBS, PCS_SEC_RNG, PCS_SEC_KEPT_IDX, PCS_SEC_KEYS = 1, 2, 3, 4
PCS_SEC_VALUES, PCS_SEC_META, PCS_SEC_K, PCS_SEC_V = 5, 6, 7, 8
PCS_KIND_MARKOV, PCS_KIND_BANK, PCS_KIND_KV = 1, 2, 3
PCS_LAYOUT_CONTIG, PCS_LAYOUT_ROWS, PCS_LAYOUT_RING = 0, 1, 2
PCS_PLACE_DEVICE, PCS_PLACE_PINNED_HOST = 0, 1
PCS_RING_START_FROM_SNAPSHOT = 0xFFFFFFFF
PCS_K_FIXED, PCS_K_BUDGET, PCS_K_FRACTION = 0, 1, 2

_DT_OF_TORCH = {
    torch.uint8: PCS_DT_U8, torch.int32: PCS_DT_I32, torch.int64: PCS_DT_I64,
    torch.float16: PCS_DT_F16, torch.bfloat16: PCS_DT_BF16, torch.float32: PCS_DT_F32,
}


class pcs_buf(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("bytes", ctypes.c_uint64),
                ("dtype", ctypes.c_uint32), ("flags", ctypes.c_uint32)]


class pcs_section(ctypes.Structure):
    _fields_ = [("type", ctypes.c_uint32), ("dtype", ctypes.c_uint32),
                ("layer", ctypes.c_uint32), ("layout", ctypes.c_uint32),
                ("base", ctypes.c_void_p), ("bytes", ctypes.c_uint64),
                ("row_bytes", ctypes.c_uint64), ("index", ctypes.c_void_p),
                ("base_rows", ctypes.c_uint64), ("ring_start", ctypes.c_uint32),
                ("window", ctypes.c_uint32), ("page_rows", ctypes.c_uint32),
                ("reserved", ctypes.c_uint32), ("dim0", ctypes.c_uint64),
                ("dim1", ctypes.c_uint64)]


class pcs_session(ctypes.Structure):
    _fields_ = [("session_id", ctypes.c_uint32), ("kind", ctypes.c_uint32),
                ("n_sections", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("sections", ctypes.POINTER(pcs_section))]


class pcs_bank(ctypes.Structure):
    _fields_ = [("keys", ctypes.c_void_p), ("query", ctypes.c_void_p),
                ("n_entries", ctypes.c_int32), ("key_dim", ctypes.c_int32),
                ("key_dtype", ctypes.c_uint32), ("reserved", ctypes.c_uint32),
                ("entry_bytes", ctypes.c_uint64)]


class pcs_prune_params(ctypes.Structure):
    _fields_ = [("rule", ctypes.c_int32), ("k_max", ctypes.c_int32),
                ("budget_bytes", ctypes.c_uint64), ("fraction", ctypes.c_double),
                ("total_bytes", ctypes.c_uint64), ("kept_align", ctypes.c_uint32),
                ("reserved", ctypes.c_uint32)]


class pcs_snapshot_info(ctypes.Structure):
    _fields_ = [("session_id", ctypes.c_uint32), ("kind", ctypes.c_uint32),
                ("n_sections", ctypes.c_int32), ("placement", ctypes.c_uint32),
                ("total_bytes", ctypes.c_uint64), ("session_fp", ctypes.c_uint64),
                ("data", ctypes.c_void_p)]


class pcs_section_info(ctypes.Structure):
    _fields_ = [("type", ctypes.c_uint32), ("dtype", ctypes.c_uint32),
                ("layer", ctypes.c_uint32), ("layout", ctypes.c_uint32),
                ("offset", ctypes.c_uint64), ("bytes", ctypes.c_uint64),
                ("fp", ctypes.c_uint64), ("dim0", ctypes.c_uint64),
                ("dim1", ctypes.c_uint64), ("aux", ctypes.c_uint64)]


class pcs_stats(ctypes.Structure):
    _fields_ = [("kernel_launches", ctypes.c_uint64), ("device_reserved", ctypes.c_uint64),
                ("host_reserved", ctypes.c_uint64), ("live_snapshots", ctypes.c_int32),
                ("sm_count", ctypes.c_int32)]


class pcs_kernel_time(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_uint64),
                ("total_ms", ctypes.c_double)]


_vp = ctypes.c_void_p
_i32 = ctypes.c_int32
_u32 = ctypes.c_uint32
_u64 = ctypes.c_uint64
_st = ctypes.c_int32

# name -> (restype, argtypes); mirrors include/pcs.h one to one.
SIGNATURES = {
    "pcs_last_error": (ctypes.c_char_p, []),
    "pcs_status_string": (ctypes.c_char_p, [_st]),
    "pcs_create": (_st, [_i32, ctypes.POINTER(_vp)]),
    "pcs_destroy": (_st, [_vp]),
    "pcs_get_stats": (_st, [_vp, ctypes.POINTER(pcs_stats)]),
    "pcs_sync": (_st, [_vp, _vp]),
    "pcs_selftest_wait": (_st, [_vp, _i32, _vp]),
    "pcs_timing_enable": (_st, [_vp, _i32]),
    "pcs_timing_read": (_st, [_vp, ctypes.POINTER(pcs_kernel_time), _i32, ctypes.POINTER(_i32)]),
    "pcs_fingerprint": (_st, [_vp, ctypes.POINTER(pcs_buf), _i32, _vp, _vp]),
    "pcs_classify": (_st, [_vp, ctypes.POINTER(pcs_buf), _i32, _vp, _vp, _vp, _vp]),
    "pcs_prune_counts": (_st, [ctypes.POINTER(pcs_bank), _i32, ctypes.POINTER(pcs_prune_params),
                               ctypes.POINTER(_i32)]),
    "pcs_prune": (_st, [_vp, ctypes.POINTER(pcs_bank), _i32, ctypes.POINTER(pcs_prune_params),
                        _vp, _vp, _vp, _vp]),
    "pcs_record_bytes": (_st, [ctypes.POINTER(pcs_section), _i32, ctypes.POINTER(_u64)]),
    "pcs_topk": (_st, [_vp, _vp, ctypes.POINTER(_i32), ctypes.POINTER(_i32), _i32, _vp, _vp, _vp]),
    "pcs_prune_global": (_st, [_vp, ctypes.POINTER(pcs_bank), _i32, _u64, _vp, _vp, _vp, _vp]),
    "pcs_budget_plan": (_st, [ctypes.POINTER(_i32), ctypes.POINTER(_u64), ctypes.POINTER(ctypes.c_double),
                              _i32, _u64, ctypes.c_double, ctypes.POINTER(_i32),
                              ctypes.POINTER(_i32), ctypes.POINTER(_i32)]),
    "pcs_checkpoint": (_st, [_vp, ctypes.POINTER(pcs_session), _i32, _u32, ctypes.POINTER(_vp),
                             _vp]),
    "pcs_fork": (_st, [_vp, _vp, ctypes.POINTER(_vp), _vp]),
    "pcs_fork_many": (_st, [_vp, ctypes.POINTER(_vp), _i32, ctypes.POINTER(_vp), _vp]),
    "pcs_restore": (_st, [_vp, ctypes.POINTER(_vp), _i32, ctypes.POINTER(pcs_session), _i32,
                          _vp]),
    "pcs_delete": (_st, [_vp, _vp]),
    "pcs_delete_many": (_st, [_vp, ctypes.POINTER(_vp), _i32]),
    "pcs_snapshot_get_info": (_st, [_vp, _vp, ctypes.POINTER(pcs_snapshot_info)]),
    "pcs_snapshot_get_section": (_st, [_vp, _vp, _i32, ctypes.POINTER(pcs_section_info)]),
    "pcs_snapshot_copy_out": (_st, [_vp, _vp, _u64, _u64, _vp, _vp]),
    "pcs_snapshot_write_file": (_st, [_vp, _vp, ctypes.c_char_p]),
    "pcs_snapshot_read_file": (_st, [_vp, ctypes.c_char_p, _u32, ctypes.POINTER(_vp)]),
    "pcs_pool_create": (_st, [_vp, _vp, _u64, _i32, ctypes.POINTER(_vp)]),
    "pcs_pool_destroy": (_st, [_vp, _vp]),
    "pcs_pool_alloc": (_st, [_vp, _vp, _vp, _i32, _vp]),
    "pcs_pool_share": (_st, [_vp, _vp, _vp, _vp, _i32, _vp]),
    "pcs_pool_prepare_write": (_st, [_vp, _vp, _vp, ctypes.c_int64, _vp, _i32, _vp]),
    "pcs_pool_release": (_st, [_vp, _vp, _vp, _i32, _vp]),
    "pcs_pool_query": (_st, [_vp, _vp, ctypes.POINTER(_i32), _vp, _vp, _vp]),
    "pcs_mismatch": (_st, [_vp, ctypes.POINTER(pcs_buf), ctypes.POINTER(pcs_buf), _i32, _vp, _vp]),
    "pcs_classify_reads": (_st, [_vp, ctypes.POINTER(pcs_buf), _i32, _vp, _vp, ctypes.c_int64, _vp,
                                 _vp]),
    "pcs_discover": (_st, [_i32, _vp, _vp, _u64, ctypes.POINTER(ctypes.c_uint8),
                           ctypes.POINTER(_i32), ctypes.POINTER(_i32)]),
    "pcs_plan_checkpoint": (_st, [_vp, ctypes.POINTER(pcs_session), _i32, _u32,
                                  ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp]),
    "pcs_plan_restore": (_st, [_vp, ctypes.POINTER(_vp), _i32, ctypes.POINTER(pcs_session), _i32,
                               ctypes.POINTER(_vp)]),
    "pcs_plan_run": (_st, [_vp, _vp, _vp]),
    "pcs_plan_destroy": (_st, [_vp, _vp]),
    "pcs_set_arena_limit": (_st, [_vp, _u32, _u64]),
    "pcs_prune_global_part": (_st, [_vp, ctypes.POINTER(pcs_bank), _i32, _u64, _u64, _vp, _vp,
                                    _vp, _vp, _vp, _vp]),
    "pcs_fingerprint_static": (_st, [ctypes.POINTER(pcs_buf), _i32, _vp, _vp]),
}
# int32 exchange(void* user, uint64_t* counts, uint64_t* bytes, int32 bins)
EXCHANGE_FN = ctypes.CFUNCTYPE(_i32, _vp, ctypes.POINTER(_u64), ctypes.POINTER(_u64), _i32)
# int32 probe(void* user, const uint8_t* keep, uint64_t* distance)
PROBE_FN = ctypes.CFUNCTYPE(_i32, _vp, ctypes.POINTER(ctypes.c_uint8), ctypes.POINTER(_u64))
PCS_STATIC_MAX_BUFFERS = 64
PCS_STATIC_MAX_NODES = 65536

_lib = None
_lock = threading.Lock()


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libpcs.so (built by ``paper_2607_21686_gb300.build``); raise if absent."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise RuntimeError(
                "libpcs.so not found at %s; build it with "
                "`python -m paper_2607_21686_gb300.build` (no CPU fallback exists)" % path)
        lib = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def budget_plan(n, entry_bytes, budget: int, fraction: float, priority=None):
    """Host shrink-then-drop plan: (k per session, shrinks, drops)."""
    lib = load_library()
    c = len(n)
    na = (ctypes.c_int32 * max(c, 1))(*n)
    eb = entry_bytes if not isinstance(entry_bytes, int) else [entry_bytes] * c
    ea = (ctypes.c_uint64 * max(c, 1))(*eb)
    pa = None if priority is None else (ctypes.c_double * max(c, 1))(*priority)
    ko = (ctypes.c_int32 * max(c, 1))()
    sh, dr = ctypes.c_int32(), ctypes.c_int32()
    check(lib.pcs_budget_plan(na, ea, pa, c, budget, fraction, ko, ctypes.byref(sh),
                              ctypes.byref(dr)), "pcs_budget_plan")
    return list(ko)[:c], sh.value, dr.value


def discover(k: int, probe, eps: int = 0):
    """Sec. 4 discovery over k components; probe(keep: list[bool]) -> D.

    Returns (PCS flags, probes run, consistent).  An exception inside the
    probe stops the procedure and is raised again here.
    """
    lib = load_library()
    failure = []

    def cb(_user, keep, dist):
        try:
            dist[0] = int(probe([bool(keep[i]) for i in range(k)]))
            return 0
        except BaseException as ex:  # re-raised below
            failure.append(ex)
            return 1

    fn = PROBE_FN(cb)
    out = (ctypes.c_uint8 * max(k, 1))()
    probes, ok = ctypes.c_int32(), ctypes.c_int32()
    st = lib.pcs_discover(k, ctypes.cast(fn, ctypes.c_void_p), None, eps, out,
                          ctypes.byref(probes), ctypes.byref(ok))
    if failure:
        raise failure[0]
    check(st, "pcs_discover")
    return [out[i] for i in range(k)], probes.value, bool(ok.value)


class PcsError(RuntimeError):
    def __init__(self, status: int, where: str):
        lib = load_library()
        self.status = status
        msg = lib.pcs_last_error().decode(errors="replace")
        name = lib.pcs_status_string(status).decode()
        super().__init__("%s failed: %s (%s)" % (where, name, msg))


def check(status: int, where: str) -> None:
    if status != PCS_OK:
        raise PcsError(status, where)


_current_raw_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream_ptr(stream) -> int:
    """The cudaStream_t of `stream` (a torch stream or an integer handle);
    None means torch's current stream on the current device, read without
    building a Stream object (a few microseconds per call otherwise)."""
    if stream is None:
        if _current_raw_stream is not None:
            return int(_current_raw_stream(torch.cuda.current_device()))
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


def _ptr(t) -> int | None:
    if t is None:
        return None
    return t.data_ptr() if t.numel() else None


def _nbytes(t: torch.Tensor) -> int:
    return t.numel() * t.element_size()


# --------------------------------------------------------------------------
# Section descriptions
# --------------------------------------------------------------------------

def contig_section(type_: int, t: torch.Tensor, layer: int = 0, dim0: int = 0, dim1: int = 0,
                   dtype: int | None = None) -> pcs_section:
    assert t.is_contiguous()
    return pcs_section(type=type_, dtype=_DT_OF_TORCH.get(t.dtype, PCS_DT_RAW) if dtype is None
                       else dtype, layer=layer, layout=PCS_LAYOUT_CONTIG, base=_ptr(t),
                       bytes=_nbytes(t), dim0=dim0, dim1=dim1)


def rows_section(type_: int, base: torch.Tensor, index: torch.Tensor, layer: int = 0,
                 dtype: int | None = None) -> pcs_section:
    """Rows index[r] of `base` (first dimension = rows)."""
    assert base.is_contiguous() and index.dtype == torch.int32 and index.is_contiguous()
    rb = _nbytes(base) // base.shape[0] if base.shape[0] else 0
    k = index.numel()
    return pcs_section(type=type_, dtype=_DT_OF_TORCH.get(base.dtype, PCS_DT_RAW) if dtype is None
                       else dtype, layer=layer, layout=PCS_LAYOUT_ROWS, base=_ptr(base),
                       bytes=rb * k, row_bytes=rb, index=_ptr(index), base_rows=base.shape[0],
                       dim0=k, dim1=rb)


def ring_section(type_: int, pool: torch.Tensor, page_table: torch.Tensor, ring_start: int,
                 window: int, layer: int = 0) -> pcs_section:
    """A paged ring window: pool [pages, page_rows, ...], page_table int32 [window/page_rows]."""
    assert pool.is_contiguous() and page_table.dtype == torch.int32 and page_table.is_contiguous()
    page_rows = pool.shape[1]
    rb = _nbytes(pool) // (pool.shape[0] * page_rows)
    return pcs_section(type=type_, dtype=_DT_OF_TORCH.get(pool.dtype, PCS_DT_RAW), layer=layer,
                       layout=PCS_LAYOUT_RING, base=_ptr(pool), bytes=rb * window, row_bytes=rb,
                       index=_ptr(page_table), base_rows=pool.shape[0],
                       ring_start=ring_start & 0xFFFFFFFF, window=window, page_rows=page_rows,
                       dim0=window, dim1=rb)


class Session:
    """A session as an ordered section list (keeps its tensors alive)."""

    def __init__(self, session_id: int, kind: int, sections, keep=()):
        self.session_id = session_id
        self.kind = kind
        self.sections = (pcs_section * len(sections))(*sections)
        self.keep = list(keep)

    def struct(self) -> pcs_session:
        return pcs_session(session_id=self.session_id, kind=self.kind,
                           n_sections=len(self.sections),
                           sections=ctypes.cast(self.sections, ctypes.POINTER(pcs_section)))


def markov_session(session_id: int, obs: torch.Tensor, rng: torch.Tensor) -> Session:
    secs = [contig_section(PCS_SEC_OBS, obs, dim0=obs.numel()),
            contig_section(PCS_SEC_RNG, rng, dim0=2, dtype=PCS_DT_U64)]
    return Session(session_id, PCS_KIND_MARKOV, secs, keep=[obs, rng])


def bank_session(session_id: int, keys: torch.Tensor, values: torch.Tensor,
                 kept: torch.Tensor) -> Session:
    """Checkpoint source: the kept rows of a bank, gathered by index."""
    secs = [contig_section(PCS_SEC_KEPT_IDX, kept, dim0=kept.numel()),
            rows_section(PCS_SEC_KEYS, keys.reshape(keys.shape[0], -1), kept),
            rows_section(PCS_SEC_VALUES, values.reshape(values.shape[0], -1), kept)]
    return Session(session_id, PCS_KIND_BANK, secs, keep=[keys, values, kept])


def bank_targets(session_id: int, kept_out: torch.Tensor, keys_out: torch.Tensor,
                 values_out: torch.Tensor) -> Session:
    """Restore target: a compacted bank holding the kept rows only."""
    k = kept_out.numel()
    secs = [contig_section(PCS_SEC_KEPT_IDX, kept_out, dim0=k),
            contig_section(PCS_SEC_KEYS, keys_out, dim0=k),
            contig_section(PCS_SEC_VALUES, values_out, dim0=k)]
    return Session(session_id, PCS_KIND_BANK, secs, keep=[kept_out, keys_out, values_out])


def kv_session(session_id: int, meta: torch.Tensor, k_pool: torch.Tensor, v_pool: torch.Tensor,
               page_table: torch.Tensor, ring_start: int, window: int,
               v_page_table: torch.Tensor = None) -> Session:
    """page_table: int32 [layers, window / page_rows] of pool page ids (of the
    K pages, and of the V pages too unless v_page_table is given)."""
    vt = page_table if v_page_table is None else v_page_table
    secs = [contig_section(PCS_SEC_META, meta, dim0=meta.numel())]
    for l in range(page_table.shape[0]):
        secs.append(ring_section(PCS_SEC_K, k_pool, page_table[l], ring_start, window, layer=l))
        secs.append(ring_section(PCS_SEC_V, v_pool, vt[l], ring_start, window, layer=l))
    return Session(session_id, PCS_KIND_KV, secs, keep=[meta, k_pool, v_pool, page_table, vt])


# --------------------------------------------------------------------------
# Context
# --------------------------------------------------------------------------

class Snapshot:
    """An opaque snapshot handle owned by a Context."""

    def __init__(self, ctx: "Context", handle: int):
        self.ctx = ctx
        self.handle = handle

    def info(self) -> pcs_snapshot_info:
        return self.ctx.info(self)

    def delete(self) -> None:
        self.ctx.delete(self)


_BUF_DTYPE = np.dtype([("ptr", np.uint64), ("bytes", np.uint64), ("dtype", np.uint32),
                       ("flags", np.uint32)])


class BufArray:
    """pcs_buf[n] describing contiguous tensors (keeps them alive)."""

    def __init__(self, tensors):
        tensors = list(tensors)
        n = len(tensors)
        a = np.zeros(max(n, 1), dtype=_BUF_DTYPE)
        if n:
            if not all(t.is_contiguous() for t in tensors):
                raise ValueError("every buffer must be contiguous")
            a["ptr"][:n] = [t.data_ptr() if t.numel() else 0 for t in tensors]
            a["bytes"][:n] = [t.numel() * t.element_size() for t in tensors]
            a["dtype"][:n] = [_DT_OF_TORCH.get(t.dtype, PCS_DT_RAW) for t in tensors]
        self.keep = tensors
        self.arr = a
        self.n = n
        self.ptr = a.ctypes.data_as(ctypes.POINTER(pcs_buf))
        self.ptr._keep = a  # the pointer keeps the array alive

    def __len__(self):
        return self.n


class Pool:
    """A copy-on-write page pool over the caller tensor `pages` ([n_pages, ...]).

    Page ids index the first dimension of `pages`; -1 is an empty slot.
    """

    def __init__(self, ctx: "Context", pages: torch.Tensor):
        assert pages.is_cuda and pages.is_contiguous() and pages.dim() >= 1
        self.ctx = ctx
        self.pages = pages
        self.n_pages = pages.shape[0]
        self.page_bytes = pages[0].numel() * pages.element_size()
        h = ctypes.c_void_p()
        check(ctx.lib.pcs_pool_create(ctx.h, pages.data_ptr(), self.page_bytes, self.n_pages,
                                      ctypes.byref(h)), "pcs_pool_create")
        self.h = h

    def alloc(self, n: int, stream=None) -> torch.Tensor:
        ids = torch.empty(n, dtype=torch.int32, device=self.pages.device)
        check(self.ctx.lib.pcs_pool_alloc(self.ctx.h, self.h, _ptr(ids), n, _stream_ptr(stream)),
              "pcs_pool_alloc")
        return ids

    def share(self, src: torch.Tensor, dst: torch.Tensor = None, stream=None) -> torch.Tensor:
        """Fork: the pages of `src` gain a holder; returns the child's table."""
        if dst is None:
            dst = torch.empty_like(src)
        check(self.ctx.lib.pcs_pool_share(self.ctx.h, self.h, _ptr(src), _ptr(dst), src.numel(),
                                          _stream_ptr(stream)), "pcs_pool_share")
        return dst

    def prepare_write(self, table: torch.Tensor, entries: torch.Tensor = None, stream=None):
        n = table.numel() if entries is None else entries.numel()
        check(self.ctx.lib.pcs_pool_prepare_write(self.ctx.h, self.h, _ptr(table), table.numel(),
                                                  _ptr(entries), n, _stream_ptr(stream)),
              "pcs_pool_prepare_write")

    def release(self, ids: torch.Tensor, stream=None):
        check(self.ctx.lib.pcs_pool_release(self.ctx.h, self.h, _ptr(ids), ids.numel(),
                                            _stream_ptr(stream)), "pcs_pool_release")

    def query(self, stream=None):
        """(free page count, holder counts uint32[n_pages], free page ids)."""
        free = ctypes.c_int32()
        counts = np.zeros(self.n_pages, dtype=np.uint32)
        ids = np.zeros(self.n_pages, dtype=np.int32)
        check(self.ctx.lib.pcs_pool_query(self.ctx.h, self.h, ctypes.byref(free),
                                          counts.ctypes.data, ids.ctypes.data,
                                          _stream_ptr(stream)), "pcs_pool_query")
        return free.value, counts, ids[:free.value].copy()

    def destroy(self):
        if self.h:
            check(self.ctx.lib.pcs_pool_destroy(self.ctx.h, self.h), "pcs_pool_destroy")
            self.h = None


class Context:
    """One libpcs context on one CUDA device."""

    def __init__(self, device: int = 0):
        self.lib = load_library()
        h = ctypes.c_void_p()
        check(self.lib.pcs_create(device, ctypes.byref(h)), "pcs_create")
        self.h = h
        self.device = device

    def close(self) -> None:
        if self.h:
            check(self.lib.pcs_destroy(self.h), "pcs_destroy")
            self.h = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def set_arena_limit(self, placement: int, nbytes: int) -> None:
        check(self.lib.pcs_set_arena_limit(self.h, placement, nbytes), "pcs_set_arena_limit")

    def stats(self) -> pcs_stats:
        s = pcs_stats()
        check(self.lib.pcs_get_stats(self.h, ctypes.byref(s)), "pcs_get_stats")
        return s

    def timing(self, on: bool) -> None:
        check(self.lib.pcs_timing_enable(self.h, 1 if on else 0), "pcs_timing_enable")

    def kernel_times(self) -> dict:
        """{kernel name: (launches, total ms)} of the launches timed so far."""
        arr = (pcs_kernel_time * 32)()
        n = ctypes.c_int32()
        check(self.lib.pcs_timing_read(self.h, arr, 32, ctypes.byref(n)), "pcs_timing_read")
        return {arr[i].name.decode(): (arr[i].launches, arr[i].total_ms)
                for i in range(min(n.value, 32))}

    def sync(self, stream=None) -> None:
        check(self.lib.pcs_sync(self.h, _stream_ptr(stream)), "pcs_sync")

    def selftest_wait(self, which: int, stream=None) -> None:
        """Enqueue the bounded-wait self-test; the next sync raises PCS_E_TIMEOUT."""
        check(self.lib.pcs_selftest_wait(self.h, which, _stream_ptr(stream)), "pcs_selftest_wait")

    # -- fingerprint / classify --------------------------------------------
    @staticmethod
    def _bufs(tensors):
        if isinstance(tensors, BufArray):
            return tensors.ptr
        return BufArray(tensors).ptr

    @staticmethod
    def buf_array(tensors) -> "BufArray":
        """A prebuilt pcs_buf array for repeated calls on the same tensors."""
        return BufArray(tensors)

    def fingerprint(self, tensors, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        n = len(tensors)
        if out is None:
            out = torch.empty(n, dtype=torch.int64, device="cuda:%d" % self.device)
        check(self.lib.pcs_fingerprint(self.h, self._bufs(tensors), n, _ptr(out),
                                       _stream_ptr(stream)), "pcs_fingerprint")
        return out

    def classify(self, tensors, fp_before: torch.Tensor, fp_after: torch.Tensor | None = None,
                 must: torch.Tensor | None = None, stream=None):
        n = len(tensors)
        dev = "cuda:%d" % self.device
        if must is None:
            must = torch.empty(n, dtype=torch.uint8, device=dev)
        if fp_after is None:
            fp_after = torch.empty(n, dtype=torch.int64, device=dev)
        check(self.lib.pcs_classify(self.h, self._bufs(tensors), n, _ptr(fp_before),
                                    _ptr(fp_after), _ptr(must), _stream_ptr(stream)),
              "pcs_classify")
        return must, fp_after

    def mismatch(self, a, b, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        """Differing bytes of each pair (a[i], b[i]), plus their length difference."""
        n = len(a)
        assert len(b) == n
        if out is None:
            out = torch.empty(n, dtype=torch.int64, device="cuda:%d" % self.device)
        check(self.lib.pcs_mismatch(self.h, self._bufs(a), self._bufs(b), n, _ptr(out),
                                    _stream_ptr(stream)), "pcs_mismatch")
        return out

    def classify_reads(self, tensors, addr: torch.Tensor, nbytes: torch.Tensor,
                       flags: torch.Tensor | None = None, stream=None) -> torch.Tensor:
        """1 for each buffer some read [addr, addr + nbytes) overlaps (state), else 0."""
        n = len(tensors)
        if flags is None:
            flags = torch.empty(n, dtype=torch.uint8, device="cuda:%d" % self.device)
        check(self.lib.pcs_classify_reads(self.h, self._bufs(tensors), n, _ptr(addr),
                                          _ptr(nbytes), addr.numel(), _ptr(flags),
                                          _stream_ptr(stream)), "pcs_classify_reads")
        return flags

    # -- prune ---------------------------------------------------------------
    @staticmethod
    def banks_array(keys_list, queries, entry_bytes):
        n = len(keys_list)
        arr = (pcs_bank * max(n, 1))()
        for s, (k, q) in enumerate(zip(keys_list, queries)):
            dt = PCS_DT_BF16 if k.dtype == torch.bfloat16 else PCS_DT_F16
            arr[s] = pcs_bank(keys=_ptr(k), query=q.data_ptr(), n_entries=k.shape[0],
                              key_dim=k.shape[1], key_dtype=dt, reserved=0,
                              entry_bytes=entry_bytes if isinstance(entry_bytes, int)
                              else entry_bytes[s])
        return arr

    @staticmethod
    def params(rule: int, k_max: int = 0, budget: int = 0, fraction: float = 0.0,
               total_bytes: int = 0, kept_align: int = 0):
        return pcs_prune_params(rule=rule, k_max=k_max, budget_bytes=budget, fraction=fraction,
                                total_bytes=total_bytes, kept_align=kept_align)

    @staticmethod
    def prune_counts(banks, n: int, params) -> list:
        """Host only: entries each bank keeps under `params`."""
        k = (ctypes.c_int32 * max(n, 1))()
        check(load_library().pcs_prune_counts(banks, n, ctypes.byref(params), k),
              "pcs_prune_counts")
        return list(k)[:n]

    def prune(self, banks, n: int, params, kept_idx: torch.Tensor, kept_off=None, scores=None,
              stream=None):
        check(self.lib.pcs_prune(self.h, banks, n, ctypes.byref(params), _ptr(scores),
                                 _ptr(kept_idx), _ptr(kept_off), _stream_ptr(stream)),
              "pcs_prune")

    @staticmethod
    def int32_array(values):
        """A ctypes int32 array (prebuilt once for repeated calls)."""
        return (ctypes.c_int32 * max(len(values), 1))(*values)

    def topk(self, keys: torch.Tensor, n, k, kept_idx: torch.Tensor, kept_off=None, stream=None):
        """Keep-k per bank by caller rank keys (CSR float32 `keys`); n and k
        are sequences of ints or prebuilt int32_array()s."""
        nb = len(n)
        na = n if isinstance(n, ctypes.Array) else self.int32_array(n)
        ka = k if isinstance(k, ctypes.Array) else self.int32_array(k)
        check(self.lib.pcs_topk(self.h, _ptr(keys), na, ka, nb, _ptr(kept_idx), _ptr(kept_off),
                                _stream_ptr(stream)), "pcs_topk")

    def prune_global(self, banks, n: int, budget: int, kept_idx: torch.Tensor,
                     kept_off: torch.Tensor, scores=None, stream=None):
        """One relevance threshold across all banks under a byte budget."""
        check(self.lib.pcs_prune_global(self.h, banks, n, budget, _ptr(scores), _ptr(kept_idx),
                                        _ptr(kept_off), _stream_ptr(stream)), "pcs_prune_global")

    def prune_global_part(self, banks, n: int, budget: int, pos_base: int, exchange,
                          kept_idx: torch.Tensor, kept_off: torch.Tensor, scores=None,
                          stream=None):
        """One part of a split population: exchange(counts, bytes) receives
        this part's per-digit histograms (numpy uint64 views) and must sum
        them over all parts in place."""
        failure = []

        def cb(_user, counts, nbytes, bins):
            try:
                c = np.ctypeslib.as_array(counts, shape=(bins,))
                b = np.ctypeslib.as_array(nbytes, shape=(bins,))
                exchange(c, b)
                return 0
            except BaseException as ex:  # re-raised below
                failure.append(ex)
                return 1

        fn = EXCHANGE_FN(cb)
        st = self.lib.pcs_prune_global_part(self.h, banks, n, budget, pos_base,
                                            ctypes.cast(fn, ctypes.c_void_p), None, _ptr(scores),
                                            _ptr(kept_idx), _ptr(kept_off), _stream_ptr(stream))
        if failure:
            raise failure[0]
        check(st, "pcs_prune_global_part")

    # -- snapshots -------------------------------------------------------------
    def record_bytes(self, session: Session) -> int:
        out = ctypes.c_uint64()
        check(self.lib.pcs_record_bytes(session.sections, len(session.sections), ctypes.byref(out)),
              "pcs_record_bytes")
        return out.value

    def checkpoint(self, sessions, placement: int = PCS_PLACE_DEVICE, stream=None) -> list:
        n = len(sessions)
        arr = (pcs_session * max(n, 1))(*[s.struct() for s in sessions])
        out = (ctypes.c_void_p * max(n, 1))()
        check(self.lib.pcs_checkpoint(self.h, arr, n, placement, out, _stream_ptr(stream)),
              "pcs_checkpoint")
        return [Snapshot(self, out[i]) for i in range(n)]

    # -- batch forms: prebuilt struct arrays, raw handle arrays ------------------
    @staticmethod
    def session_array(sessions):
        """A ctypes pcs_session array for repeated batch calls (keeps `sessions`)."""
        arr = (pcs_session * max(len(sessions), 1))(*[s.struct() for s in sessions])
        arr._keep = list(sessions)
        return arr

    def checkpoint_raw(self, arr, n: int, placement: int = PCS_PLACE_DEVICE, stream=None):
        """checkpoint of a prebuilt session array; returns a ctypes handle array."""
        out = (ctypes.c_void_p * max(n, 1))()
        check(self.lib.pcs_checkpoint(self.h, arr, n, placement, out, _stream_ptr(stream)),
              "pcs_checkpoint")
        return out

    def fork_raw(self, handles, n: int, stream=None):
        """fork of n snapshots in one call; returns a ctypes handle array."""
        out = (ctypes.c_void_p * max(n, 1))()
        check(self.lib.pcs_fork_many(self.h, handles, n, out, _stream_ptr(stream)), "pcs_fork_many")
        return out

    def restore_raw(self, handles, n: int, arr, verify: int = 0, stream=None) -> None:
        check(self.lib.pcs_restore(self.h, handles, n, arr, verify, _stream_ptr(stream)),
              "pcs_restore")

    def delete_raw(self, handles, n: int) -> None:
        check(self.lib.pcs_delete_many(self.h, handles, n), "pcs_delete_many")

    # -- prepared calls ---------------------------------------------------------
    def plan_checkpoint(self, arr, n: int, placement: int = PCS_PLACE_DEVICE, stream=None):
        """Plan checkpoint(s) of a prebuilt session array and run it once:
        (plan handle, ctypes array of the n snapshot handles)."""
        out = (ctypes.c_void_p * max(n, 1))()
        plan = ctypes.c_void_p()
        check(self.lib.pcs_plan_checkpoint(self.h, arr, n, placement, out, ctypes.byref(plan),
                                           _stream_ptr(stream)), "pcs_plan_checkpoint")
        return plan, out

    def plan_restore(self, handles, n: int, arr, verify: int = 0):
        plan = ctypes.c_void_p()
        check(self.lib.pcs_plan_restore(self.h, handles, n, arr, verify, ctypes.byref(plan)),
              "pcs_plan_restore")
        return plan

    def plan_run(self, plan, stream=None) -> None:
        check(self.lib.pcs_plan_run(self.h, plan, _stream_ptr(stream)), "pcs_plan_run")

    def plan_destroy(self, plan) -> None:
        check(self.lib.pcs_plan_destroy(self.h, plan), "pcs_plan_destroy")

    def fork(self, snap: Snapshot, stream=None) -> Snapshot:
        out = ctypes.c_void_p()
        check(self.lib.pcs_fork(self.h, snap.handle, ctypes.byref(out), _stream_ptr(stream)),
              "pcs_fork")
        return Snapshot(self, out.value)

    def restore(self, snaps, targets, verify=False, stream=None) -> None:
        """verify: False/0 none, True/1 check and wait, 2 check, report at sync."""
        n = len(snaps)
        hs = (ctypes.c_void_p * max(n, 1))(*[s.handle for s in snaps])
        arr = (pcs_session * max(n, 1))(*[t.struct() for t in targets])
        check(self.lib.pcs_restore(self.h, hs, n, arr, int(verify), _stream_ptr(stream)),
              "pcs_restore")

    def restore_status(self, snaps, targets, verify: bool = True, stream=None) -> int:
        n = len(snaps)
        hs = (ctypes.c_void_p * max(n, 1))(*[s.handle for s in snaps])
        arr = (pcs_session * max(n, 1))(*[t.struct() for t in targets])
        return self.lib.pcs_restore(self.h, hs, n, arr, 1 if verify else 0, _stream_ptr(stream))

    def delete(self, snap: Snapshot) -> None:
        check(self.lib.pcs_delete(self.h, snap.handle), "pcs_delete")
        snap.handle = None

    def info(self, snap: Snapshot) -> pcs_snapshot_info:
        out = pcs_snapshot_info()
        check(self.lib.pcs_snapshot_get_info(self.h, snap.handle, ctypes.byref(out)),
              "pcs_snapshot_get_info")
        return out

    def section(self, snap: Snapshot, i: int) -> pcs_section_info:
        out = pcs_section_info()
        check(self.lib.pcs_snapshot_get_section(self.h, snap.handle, i, ctypes.byref(out)),
              "pcs_snapshot_get_section")
        return out

    def record(self, snap: Snapshot, stream=None) -> torch.Tensor:
        """A host copy of the whole record (uint8)."""
        nb = self.info(snap).total_bytes
        out = torch.empty(nb, dtype=torch.uint8, pin_memory=True)
        self.copy_out(snap, 0, nb, out, stream)
        torch.cuda.current_stream().synchronize() if stream is None else stream.synchronize()
        return out

    def copy_out(self, snap: Snapshot, offset: int, nbytes: int, dst: torch.Tensor, stream=None):
        check(self.lib.pcs_snapshot_copy_out(self.h, snap.handle, offset, nbytes, dst.data_ptr(),
                                             _stream_ptr(stream)), "pcs_snapshot_copy_out")

    def write_file(self, snap: Snapshot, path: str) -> None:
        check(self.lib.pcs_snapshot_write_file(self.h, snap.handle, path.encode()),
              "pcs_snapshot_write_file")

    def read_file(self, path: str, placement: int = PCS_PLACE_DEVICE) -> Snapshot:
        out = ctypes.c_void_p()
        check(self.lib.pcs_snapshot_read_file(self.h, path.encode(), placement, ctypes.byref(out)),
              "pcs_snapshot_read_file")
        return Snapshot(self, out.value)
