"""The committed-length bookkeeping of the asynchronous fast-slow session (Sec. 3.3:
ticks read the cache as it stands while appends run behind them), checked on the CPU:
the product header ``csrc/ledger.h`` is compiled with a randomised schedule driver
(``tests/cpp/ledger_check.cpp``) and every tick's snapshot must hold exactly the rows
of completed appends, never a row being written."""
from __future__ import annotations

import os
import shutil
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_15621_gb300", "csrc")


@pytest.mark.skipif(shutil.which("g++") is None, reason="needs a host C++ compiler")
def test_snapshots_never_include_rows_in_flight():
    with tempfile.TemporaryDirectory() as tmp:
        exe = os.path.join(tmp, "ledger_check")
        subprocess.run(["g++", "-std=c++17", "-O1", "-I", CSRC, os.path.join(ROOT, "tests", "cpp", "ledger_check.cpp"),
                        "-o", exe], check=True, capture_output=True, text=True)
        res = subprocess.run([exe, "300"], capture_output=True, text=True, timeout=120)
    assert res.returncode == 0, res.stdout + res.stderr
    assert res.stdout.startswith("ok ") and int(res.stdout.split()[1]) > 10000
