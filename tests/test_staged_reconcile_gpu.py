"""The reconcile with its rows staged through shared memory by bulk copies
(cpdp_set_reconcile_staging, the measured alternative to direct loads): parity
with the oracle at the ResNet-50 shape, bit-identical results to the default
reconcile at every worker count, ragged tile and slot count it accepts, the
settings it refuses, and no bounded wait running out. Also the plain
streaming floor kernel the benchmark compares small launches with."""
import numpy as np
import pytest
import torch

from paper_2607_21224_gb300 import cpdp
from paper_2607_21224_gb300 import workloads as wls
from paper_2607_21224_gb300.state import CPDPState
from parity import run_and_check, windows

pytestmark = pytest.mark.gpu

HYPER = dict(lr=0.1, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5)


def _run(W, N, stages, steps=4, alpha=1.0, seed=5):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(seed)
    theta0 = torch.randn(N, device=dev, generator=gen) * 0.05
    grads = [torch.randn(W, N, device=dev, generator=gen) * 1e-3 for _ in range(steps)]
    with CPDPState(W, N, alpha=alpha, **HYPER) as st:
        st.init_params(theta0)
        st.set_reconcile_staging(stages)
        for t in range(1, steps + 1):
            st.step(grads[t - 1], t, steps)
        torch.cuda.synchronize()
        timeouts = st.wait_timeouts()
        return [x.clone() for x in (st.params, st.mom, st.anchor, st.slow_v)], timeouts


@pytest.mark.parametrize("W", [1, 2, 3, 5, 8, 16])
@pytest.mark.parametrize("N", [4, 512, 4 * (512 * 3 + 7), 4 * 152 * 512 + 8])
def test_staged_reconcile_bit_identical_to_direct_loads(W, N):
    want, _ = _run(W, N, 0)
    for stages in (2, 4, 8):
        try:
            got, timeouts = _run(W, N, stages)
        except cpdp.CPDPError as e:  # too many slots of (3W + 2) 2 KB segments for a block's shared memory
            assert e.status == cpdp.CPDP_EINVAL and "shared memory" in str(e)
            assert stages * (3 * W + 2) * 2048 > 200 * 1024
            continue
        assert timeouts == 0
        for a, b in zip(got, want):
            assert torch.equal(a.view(torch.int32), b.view(torch.int32)), (W, N, stages)


def test_staged_reconcile_parity_resnet50():
    """The full ResNet-50/CIFAR-100 shape (W = 8, K = 4) through one epoch,
    sampled columns against the oracle, replicas bit-identical after every
    reconcile."""
    wl = wls.resnet50_cifar100()
    run_and_check(wl, cols=windows(wl, width=1024, n_random=1024, boundaries=6), steps=8, staging=4)


def test_staged_reconcile_refuses_what_it_does_not_cover():
    dev = torch.device("cuda")
    W, N = 4, 4 * 1024
    g = torch.randn(W, N, device=dev) * 1e-3
    with CPDPState(W, N, **HYPER) as st:
        st.init_params(torch.zeros(N, device=dev))
        for bad in (1, 9, -1):
            with pytest.raises(cpdp.CPDPError) as e:
                st.set_reconcile_staging(bad)
            assert e.value.status == cpdp.CPDP_EINVAL
        st.set_reconcile_staging(2)
        for setup in (lambda: st.set_method("localsgd"), lambda: st.set_state_reconcile(True),
                      lambda: st.set_method("ddp")):
            setup()
            with pytest.raises(cpdp.CPDPError) as e:
                st.reconcile(g)
            assert e.value.status == cpdp.CPDP_ESTATE and "staged" in str(e.value)
            st.set_method("cpdp")
            st.set_state_reconcile(False)
        with pytest.raises(cpdp.CPDPError) as e:
            st.reconcile(g.to(torch.bfloat16))
        assert e.value.status == cpdp.CPDP_ESTATE
        st.reconcile(g)  # supported settings run
        st.set_adamw()
        with pytest.raises(cpdp.CPDPError) as e:
            st.reconcile(g)
        assert e.value.status == cpdp.CPDP_ESTATE
        torch.cuda.synchronize()
        assert st.wait_timeouts() == 0
    with CPDPState(17, 64, **HYPER) as st:
        with pytest.raises(cpdp.CPDPError) as e:
            st.set_reconcile_staging(2)
        assert e.value.status == cpdp.CPDP_EINVAL and "16" in str(e.value)
    with CPDPState(2, 66, **HYPER) as st:
        with pytest.raises(cpdp.CPDPError) as e:
            st.set_reconcile_staging(2)
        assert e.value.status == cpdp.CPDP_EINVAL and "multiple of 4" in str(e.value)


@pytest.mark.parametrize("grid", [0, 3])
def test_floor_stream_writes_the_sum_of_its_rows(grid):
    dev = torch.device("cuda")
    n = 4 * 1000 + 4
    ins = [torch.full((n,), float(k + 1), device=dev) for k in range(5)]
    outs = [torch.empty(n, device=dev) for _ in range(3)]
    cpdp.cpdp_floor_stream(ins, outs, n, grid, torch.cuda.current_stream().cuda_stream)
    cpdp.cpdp_floor_empty(7, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    for o in outs:
        assert torch.equal(o, torch.full((n,), 15.0, device=dev))
    # in place over its own inputs, as the benchmark runs it
    cpdp.cpdp_floor_stream(ins[:2], ins[:2], n, grid, torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    assert np.all(ins[0].cpu().numpy() == 3.0) and np.all(ins[1].cpu().numpy() == 3.0)


def test_bounded_waits_end_a_launch_whose_loads_never_come():
    """The staged reconcile's waits are bounded: with one tile's loads withheld,
    the warps waiting for it give up (counted by cpdp_wait_timeouts), the launch
    ends after a few seconds, every other tile is reconciled as usual, and the
    context keeps working."""
    import time
    dev = torch.device("cuda")
    W, N, tile = 4, 4 * 1024, 3  # 8 tiles of 512 columns
    gen = torch.Generator(device=dev).manual_seed(21)
    theta0 = torch.randn(N, device=dev, generator=gen) * 0.05
    g = torch.randn(W, N, device=dev, generator=gen) * 1e-3
    with CPDPState(W, N, **HYPER) as ref, CPDPState(W, N, **HYPER) as st:
        for x in (ref, st):
            x.init_params(theta0)
            x.set_reconcile_staging(2)
            x.local_step(g)
        ref.reconcile(g)
        st.wait_timeouts()  # start from zero
        cpdp.cpdp_withhold_staged_tile(st.ctx, tile)
        t0 = time.time()
        st.reconcile(g)
        torch.cuda.synchronize()
        elapsed = time.time() - t0
        assert st.wait_timeouts() > 0 and 1.5 < elapsed < 60
        keep = torch.ones(N, dtype=torch.bool, device=dev)
        keep[tile * 512:(tile + 1) * 512] = False
        for a, b in ((st.params, ref.params), (st.mom, ref.mom), (st.anchor, ref.anchor), (st.slow_v, ref.slow_v)):
            assert torch.equal(a[..., keep], b[..., keep])
        st.init_params(theta0)  # the context keeps working, and the hook applied to one launch only
        st.local_step(g)
        st.reconcile(g)
        torch.cuda.synchronize()
        assert st.wait_timeouts() == 0
        for a, b in ((st.params, ref.params), (st.anchor, ref.anchor)):
            assert torch.equal(a, b)
