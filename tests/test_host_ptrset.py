"""Host: the session table's set of live snapshot handles (pcs::PtrSet, an
open-addressed pointer set) against std::unordered_set, over random
inserts, erases, membership tests of values never inserted, reserve and
clear (tests/host/ptrset_check.cpp, built here with g++)."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_21686_gb300", "csrc")


@pytest.fixture(scope="module")
def checker(tmp_path_factory):
    gxx = shutil.which("g++")
    if not gxx:
        pytest.skip("no g++")
    exe = str(tmp_path_factory.mktemp("ptrset") / "ptrset_check")
    subprocess.run([gxx, "-O2", "-std=c++17", "-I", CSRC,
                    os.path.join(ROOT, "tests", "host", "ptrset_check.cpp"), "-o", exe], check=True)
    return exe


@pytest.mark.parametrize("seed", [1, 2, 3, 4])
def test_ptrset_matches_unordered_set(checker, seed):
    out = subprocess.run([checker, str(seed), "300000"], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0 and out.stdout.strip() == "ok", out.stdout + out.stderr
