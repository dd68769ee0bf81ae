"""The C-ABI library builds, loads and exports every declared symbol (CPU).

Also checks, without a GPU, the host-only entry points against the oracle
(k-rules, record sizes) and that the ctypes mirror of every struct has the
layout the C compiler gives include/pcs.h.
"""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import build as pcs_build
from paper_2607_21686_gb300 import pcs

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pcs.h")


@pytest.fixture(scope="module")
def lib():
    pcs_build.build()
    return pcs.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(pcs_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 20
    for n in names:
        assert hasattr(lib, n), n
    # The binding mirrors exactly the declared functions.
    assert sorted(pcs.SIGNATURES) == names


def test_exported_symbols_via_nm(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", pcs.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (pcs_[a-z_]+)\b", out))
    assert set(declared_functions()) <= exported


_LAYOUT_PROBE = r"""
#include <stddef.h>
#include <stdio.h>
#include "pcs.h"
#define S(T) printf(#T " %zu\n", sizeof(T));
#define O(T, f) printf(#T "." #f " %zu\n", offsetof(T, f));
int main(void) {
  S(pcs_buf) O(pcs_buf, bytes) O(pcs_buf, dtype)
  S(pcs_section) O(pcs_section, base) O(pcs_section, bytes) O(pcs_section, index)
  O(pcs_section, base_rows) O(pcs_section, ring_start) O(pcs_section, dim0) O(pcs_section, dim1)
  S(pcs_session) O(pcs_session, n_sections) O(pcs_session, sections)
  S(pcs_bank) O(pcs_bank, n_entries) O(pcs_bank, key_dtype) O(pcs_bank, entry_bytes)
  S(pcs_prune_params) O(pcs_prune_params, budget_bytes) O(pcs_prune_params, fraction)
  O(pcs_prune_params, total_bytes) O(pcs_prune_params, kept_align)
  S(pcs_snapshot_info) O(pcs_snapshot_info, total_bytes) O(pcs_snapshot_info, data)
  S(pcs_section_info) O(pcs_section_info, offset) O(pcs_section_info, aux)
  S(pcs_stats) O(pcs_stats, live_snapshots)
  S(pcs_kernel_time) O(pcs_kernel_time, launches) O(pcs_kernel_time, total_ms)
  return 0;
}
"""


def test_ctypes_structs_match_header(tmp_path):
    src = tmp_path / "probe.c"
    exe = tmp_path / "probe"
    src.write_text(_LAYOUT_PROBE)
    subprocess.run(["gcc", "-std=c11", "-I", os.path.dirname(HEADER), "-o", str(exe), str(src)],
                   check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout
    for line in out.strip().splitlines():
        name, val = line.split()
        val = int(val)
        if "." in name:
            t, f = name.split(".")
            assert getattr(getattr(pcs, t), f).offset == val, name
        else:
            assert ctypes.sizeof(getattr(pcs, name)) == val, name


def test_status_strings(lib):
    assert lib.pcs_status_string(pcs.PCS_E_CORRUPT) == b"PCS_E_CORRUPT"
    assert lib.pcs_status_string(pcs.PCS_OK) == b"PCS_OK"


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU error path")
def test_create_without_gpu_fails_loudly(lib):
    h = ctypes.c_void_p()
    st = lib.pcs_create(0, ctypes.byref(h))
    assert st == pcs.PCS_E_CUDA
    assert b"CUDA" in lib.pcs_last_error() or lib.pcs_last_error()


def test_selftest_wait_rejects_a_null_context(lib):
    assert lib.pcs_selftest_wait(None, 0, None) == pcs.PCS_E_INVAL


def _banks(n_list, entry_bytes):
    arr = (pcs.pcs_bank * len(n_list))()
    for i, n in enumerate(n_list):
        arr[i] = pcs.pcs_bank(keys=None, query=None, n_entries=n, key_dim=8,
                              key_dtype=pcs.PCS_DT_F16, entry_bytes=entry_bytes)
    return arr


def _counts(lib, n_list, params, entry_bytes=3072):
    k = (ctypes.c_int32 * len(n_list))()
    st = lib.pcs_prune_counts(_banks(n_list, entry_bytes), len(n_list), ctypes.byref(params), k)
    assert st == 0, lib.pcs_last_error()
    return list(k)


@pytest.mark.parametrize("seed", range(5))
def test_prune_counts_match_oracle(lib, seed):
    rnd = np.random.default_rng(seed)
    n = rnd.integers(0, 5000, 300).astype(np.int32)
    E = 3072
    total = int(n.astype(np.int64).sum()) * E
    for B in [total // 3, total // 2, total, total * 2, 8 << 30]:
        p = pcs.pcs_prune_params(rule=pcs.PCS_K_BUDGET, budget_bytes=B)
        assert _counts(lib, n.tolist(), p, E) == oracle.k_budget(n, E, B).tolist()
    for kmax in [0, 1, 128, 10**6]:
        p = pcs.pcs_prune_params(rule=pcs.PCS_K_FIXED, k_max=kmax)
        assert _counts(lib, n.tolist(), p) == oracle.k_fixed(n, kmax).tolist()
    for frac in [0.0, 0.04, 0.12, 0.25, 0.5, 0.627, 1.0]:
        p = pcs.pcs_prune_params(rule=pcs.PCS_K_FRACTION, fraction=frac)
        assert _counts(lib, n.tolist(), p) == oracle.k_fraction(n, frac).tolist()


def test_prune_counts_rejects_bad_params(lib):
    p = pcs.pcs_prune_params(rule=7)
    k = (ctypes.c_int32 * 1)()
    assert lib.pcs_prune_counts(_banks([3], 1), 1, ctypes.byref(p), k) == pcs.PCS_E_INVAL
    p = pcs.pcs_prune_params(rule=pcs.PCS_K_FRACTION, fraction=1.5)
    assert lib.pcs_prune_counts(_banks([3], 1), 1, ctypes.byref(p), k) == pcs.PCS_E_INVAL
    # A whole-population T smaller than these banks' own bytes cannot be right.
    p = pcs.pcs_prune_params(rule=pcs.PCS_K_BUDGET, budget_bytes=1, total_bytes=2)
    assert lib.pcs_prune_counts(_banks([3], 1), 1, ctypes.byref(p), k) == pcs.PCS_E_INVAL


def test_budget_counts_of_a_part_use_the_whole_population(lib):
    # Counts of a part of the banks with the whole population's T equal the
    # whole population's counts for those banks (the sharded budget rule).
    rnd = np.random.default_rng(9)
    n = rnd.integers(0, 5000, 400).astype(np.int32)
    E = 3072
    T = int(n.astype(np.int64).sum()) * E
    for B in (T // 7, T // 2, T - 1, T):
        want = oracle.k_budget(n, E, B).tolist()
        for part in (slice(0, 150), slice(150, 400), slice(None, None, 3)):
            p = pcs.pcs_prune_params(rule=pcs.PCS_K_BUDGET, budget_bytes=B, total_bytes=T)
            assert _counts(lib, n[part].tolist(), p, E) == want[part]
        p = pcs.pcs_prune_params(rule=pcs.PCS_K_BUDGET, budget_bytes=B, total_bytes=T)
        assert _counts(lib, n.tolist(), p, E) == want


def test_record_bytes_match_oracle(lib):
    rnd = np.random.default_rng(3)
    for _ in range(50):
        ns = int(rnd.integers(1, 60))
        sizes = rnd.integers(0, 100000, ns)
        arr = (pcs.pcs_section * ns)()
        sp = oracle.SessionSpec(0, 0)
        keep = []
        for i, b in enumerate(sizes.tolist()):
            arr[i] = pcs.pcs_section(layout=pcs.PCS_LAYOUT_CONTIG, bytes=b)
            a = np.zeros(b, np.uint8)
            keep.append(a)
            sp.contig(1, 1, a)
        out = ctypes.c_uint64()
        assert lib.pcs_record_bytes(arr, ns, ctypes.byref(out)) == 0
        assert out.value == oracle.record_bytes(sp)


@pytest.mark.parametrize("seed", range(10))
def test_budget_plan_matches_oracle(lib, seed):
    rnd = np.random.default_rng(100 + seed)
    S = int(rnd.integers(1, 300))
    n = rnd.integers(0, 500, S).tolist()
    E = rnd.integers(1, 4096, S).tolist()
    pr = rnd.normal(size=S).tolist() if seed % 2 else None
    total = sum(a * b for a, b in zip(n, E))
    for B in [total + 1, total, total * 3 // 4, total // 4, total // 50, 0]:
        for frac in [0.0, 0.12, 0.5]:
            got = pcs.budget_plan(n, E, B, frac, priority=pr)
            k, sh, dr = oracle.budget_plan(n, E, B, frac, priority=pr)
            assert got == (k.tolist(), sh, dr), (B, frac)
