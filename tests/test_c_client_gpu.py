"""The C ABI used from plain C (tests/abi_c/cpdp_c_client.c): compiled with nvcc
against include/cpdp.h and libcpdp.so, it runs the hand-derived worked
examples, with gradients in device memory or fed from page-locked host memory
through cpdp_step_host, and with the reconcile's staged and warp-shuffle
variants, and must reproduce them bit for bit (the examples are exact in
float32, so every summation order gives the same bits); it also reads back
which reconcile kernel ran."""
import subprocess

import numpy as np
import pytest

from oracle_pins import GOLDEN_CASES, load_golden
from paper_2607_21224_gb300 import build

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def client(tmp_path_factory):
    lib = build.build_library()
    src = build.ROOT / "tests" / "abi_c" / "cpdp_c_client.c"
    exe = tmp_path_factory.mktemp("c_client") / "cpdp_c_client"
    subprocess.run([build.nvcc_path(), "-x", "cu", *build.ARCH, f"-I{build.INCLUDE}", "-o", str(exe), str(src),
                    f"-L{lib.parent}", "-lcpdp", f"-Xlinker=-rpath={lib.parent}"], check=True)
    return exe


@pytest.mark.parametrize("mode", ["device", "host", "staged", "shuffle"])
@pytest.mark.parametrize("name", GOLDEN_CASES)
def test_c_client_reproduces_golden(client, name, mode):
    c = load_golden(name)
    vals = [c["W"], c["N"], c["K"], c["T"], c["lr"], c["momentum"], c["weight_decay"], c["beta"], c["alpha"]]
    vals += c["theta0"] + [x for step in c["grads"] for row in step for x in row]
    out = subprocess.run([str(client), mode], input=" ".join(map(str, vals)), capture_output=True, text=True,
                         check=True)
    lines = out.stdout.strip().splitlines()
    W = c["W"]
    per_step = 1 + 2 * W + 2
    for k, want in enumerate(c["after"]):
        block = lines[k * per_step:(k + 1) * per_step]
        t, synced = map(int, block[0].split())
        assert (t, bool(synced)) == (want["t"], want["sync"])
        rows = [np.array(list(map(float, ln.split()))) for ln in block[1:]]
        assert np.array_equal(np.stack(rows[:W]), np.array(want["theta"]))
        assert np.array_equal(np.stack(rows[W:2 * W]), np.array(want["buf"]))
        assert np.array_equal(rows[2 * W], np.array(want["theta_ref"]))
        assert np.array_equal(rows[2 * W + 1], np.array(want["v"]))
    # the kernel the last reconcile launched, as cpdp_reconcile_kernel reports it
    assert lines[-1].startswith("kernel ")
    kernel = lines[-1].split()[1]
    if mode == "staged":
        assert kernel == "reconcile_tma_kernel"
    elif mode == "shuffle":
        assert kernel == "reconcile_shuffle_kernel"
    else:
        want_kernel = "reconcile_scalar_kernel" if c["N"] % 4 else None
        assert kernel in ("reconcile_vec4_kernel", "reconcile_onepass_kernel", "reconcile_scalar_kernel")
        assert want_kernel is None or kernel == want_kernel
