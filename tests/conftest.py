"""Shared pytest set-up: import paths, the `gpu` marker, and built libraries."""
from __future__ import annotations

import sys
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]
for p in (str(ROOT), str(ROOT / "tests")):
    if p not in sys.path:
        sys.path.insert(0, p)

# test_abi_fuzz.py holds host-only, property-based tests that need hypothesis.
# Where hypothesis is not installed the module is left out of collection
# instead of being reported as one skipped item.
try:
    import hypothesis  # noqa: F401
except ImportError:
    collect_ignore = ["test_abi_fuzz.py"]


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (built for GB300, sm_103a)")


def pytest_collection_modifyitems(config, items):
    # Without a visible GPU the gpu-marked tests cannot run at all; they are
    # reported as skipped rather than erroring. On a GPU machine they run.
    import torch

    if torch.cuda.is_available():
        return
    skip = pytest.mark.skip(reason="no CUDA device visible")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


@pytest.fixture(scope="session", autouse=True)
def _libraries_built():
    """Compile libcpdp.so (nvcc, sm_103a) and the oracle if missing or stale, so
    the tests always exercise the current sources. A no-op when up to date."""
    from paper_2607_21224_gb300 import build
    import oracle

    build.build_library()
    oracle.build_oracle()


@pytest.fixture(scope="session")
def oracle_lib():
    import oracle

    return oracle.default()
