"""Randomised GPU parity: seeded random configurations of the whole path
(worker count, size including the scalar path's odd N, tensor split, K, epoch
length, method, optimizer, state reconciliation, gradient type and every
hyperparameter), each run through an epoch on the GPU and on the fp64 oracle
with every state array compared after every step (the tolerance and replica
checks of tests/parity.py). The configurations come from a fixed seed, so a
failure names a reproducible case."""
import random

import pytest

from paper_2607_21224_gb300 import workloads as wls
from parity import run_and_check

pytestmark = pytest.mark.gpu


def _case(i: int) -> tuple[wls.Workload, str, bool]:
    rng = random.Random(1000 + i)
    W = rng.choice([1, 2, 3, 4, 5, 8, 9, 16, 31, 40])
    N = rng.choice([rng.randrange(1, 64), 4 * rng.randrange(1, 12000), rng.randrange(1, 40000)])
    K = rng.randrange(1, 6)
    T = rng.randrange(K, 3 * K + 2)
    method = rng.choice(["cpdp", "cpdp", "localsgd", "ddp"])
    opt = rng.choice(["sgd", "sgd", "adamw"])
    state_sync = method != "ddp" and rng.random() < 0.3
    kw = dict(grad_dtype=rng.choice(["f32", "bf16"]), beta=rng.choice([0.0, 0.3, 0.5, 0.7, 0.9]),
              alpha=rng.choice([1.0, 1.0, 0.5, 1.5]), grad_std=rng.choice([1e-3, 1e-2]),
              heavy_tail_p=rng.choice([0.0, 0.0, 0.01]))
    if opt == "adamw":
        kw.update(lr=rng.choice([1e-4, 5e-4, 1e-3]), weight_decay=rng.choice([0.0, 0.05]), momentum=0.0,
                  optimizer="adamw", adam_beta1=rng.choice([0.9, 0.8]), adam_beta2=rng.choice([0.999, 0.95]))
    else:
        kw.update(lr=rng.choice([0.01, 0.1, 0.4]), momentum=rng.choice([0.0, 0.5, 0.9]),
                  weight_decay=rng.choice([0.0, 5e-4, 1e-2]))
    tensors = min(N, rng.randrange(1, 6))
    wl = wls.Workload(f"rand{i}", W=W, tensors=tuple(wls.flat_tensors(N, tensors, 0.05)), K=K, T=T, **kw)
    return wl, method, state_sync


@pytest.mark.parametrize("i", range(500))
def test_random_configuration(i):
    wl, method, state_sync = _case(i)
    run_and_check(wl, method=method, state_sync=state_sync)
