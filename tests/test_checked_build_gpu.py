"""The index-checked debug build (libcpdp_checked.so, compiled with
-DCPDP_CHECKED): every kernel compares each global-memory index with the extent
of the buffer it addresses and counts any outside it. Every kernel variant runs
through it (tests/checked_scenarios.py, in a process of its own), must count no
out-of-range index, and must give results bit-identical to the release library
on the same inputs, which in turn reports -1 (no checks compiled in). With
compute-sanitizer closed on this pool, this is the check that the kernels stay
inside their buffers at every size, worker count and variant tested."""
import json
import os
import subprocess
import sys
from pathlib import Path

import pytest

from paper_2607_21224_gb300 import build

pytestmark = pytest.mark.gpu

SCENARIOS = Path(__file__).resolve().parent / "checked_scenarios.py"


def _run(library: Path | None) -> dict:
    env = dict(os.environ)
    env.pop("CPDP_LIBRARY", None)
    if library is not None:
        env["CPDP_LIBRARY"] = str(library)
    proc = subprocess.run([sys.executable, str(SCENARIOS)], env=env, capture_output=True, text=True, timeout=600)
    assert proc.returncode == 0, proc.stderr[-3000:]
    return json.loads(proc.stdout.strip().splitlines()[-1])


def test_checked_build_counts_no_bad_index_and_matches_release():
    checked_lib = build.build_library(checked=True)
    release = _run(None)
    checked = _run(checked_lib)
    assert release["library"] == "libcpdp.so" and checked["library"] == "libcpdp_checked.so"
    assert set(release["bad"].values()) == {-1}
    assert all(v == 0 for v in checked["bad"].values()), {k: v for k, v in checked["bad"].items() if v}
    assert checked["digests"] == release["digests"]
    assert len(release["digests"]) == 5 * 2 * 2 * 2 * 7 + 6 + 4 + 2
