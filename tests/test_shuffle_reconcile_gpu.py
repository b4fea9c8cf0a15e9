"""The reconcile with the worker rows split across a warp's lanes and the
W-way sums finished with warp shuffles (cpdp_set_reconcile_shuffle, the
measured alternative to per-thread register sums): parity with the oracle at
the ResNet-50 shape and at small ragged sizes, replicas bit-identical, the
same bits as the default reconcile up to three workers and the same values to
rounding beyond, and the settings it refuses."""
import numpy as np
import pytest
import torch

from paper_2607_21224_gb300 import cpdp
from paper_2607_21224_gb300 import workloads as wls
from paper_2607_21224_gb300.state import CPDPState
from parity import TOL, run_and_check, scaled_error, windows

pytestmark = pytest.mark.gpu

HYPER = dict(lr=0.1, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5)


def _run(W, N, shuffle, steps=4):
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(9)
    theta0 = torch.randn(N, device=dev, generator=gen) * 0.05
    grads = [torch.randn(W, N, device=dev, generator=gen) * 1e-3 for _ in range(steps)]
    with CPDPState(W, N, **HYPER) as st:
        st.init_params(theta0)
        st.set_reconcile_shuffle(shuffle)
        for t in range(1, steps + 1):
            st.step(grads[t - 1], t, steps)
        torch.cuda.synchronize()
        p = st.params.view(torch.int32)
        assert torch.equal(p, p[0:1].expand_as(p)) and torch.equal(p[0], st.anchor.view(torch.int32))
        return [x.clone() for x in (st.params, st.mom, st.anchor, st.slow_v)]


@pytest.mark.parametrize("W", [1, 2, 3, 4, 5, 8, 13, 16, 32])
@pytest.mark.parametrize("N", [4, 4 * 7, 4 * (256 * 3 + 5)])
def test_shuffle_reconcile_matches_register_sums(W, N):
    """Up to three workers the partial sums add in worker order: the same bits
    as the default. Beyond, the parameters and theta_ref agree to 1e-5 of their
    own size and v to 1e-5 in parameter units (v is a difference of two
    parameter-sized numbers); every array is checked against the oracle in the
    parity tests below."""
    want = _run(W, N, False)
    got = _run(W, N, True)
    if W <= 3:
        for a, b in zip(got, want):
            assert torch.equal(a.view(torch.int32), b.view(torch.int32))
        return
    host = lambda x: x.double().cpu().numpy()  # noqa: E731
    tid = np.zeros(N, dtype=np.int64)
    assert scaled_error(host(got[0]), host(want[0]), tid) <= TOL
    assert scaled_error(host(got[2]), host(want[2]), tid) <= TOL
    assert scaled_error(host(got[3]), host(want[3]), tid, scale=host(want[2])) <= TOL


@pytest.mark.parametrize("W", [4, 5, 8, 13, 16, 32])
@pytest.mark.parametrize("N", [4 * 7, 4 * (256 * 3 + 5)])
def test_shuffle_reconcile_parity_small(W, N):
    """Every state array against the oracle after every step, two epochs'
    worth of reconciles (the tolerance reading of tests/parity.py)."""
    wl = wls.Workload(f"shuffle_{W}_{N}", W=W, tensors=tuple(wls.flat_tensors(N, 2, 0.05)), K=2, T=6)
    run_and_check(wl, shuffle=True)


def test_shuffle_reconcile_parity_resnet50():
    """The full ResNet-50/CIFAR-100 shape (W = 8, K = 4), sampled columns
    against the oracle, replicas bit-identical after every reconcile; the
    no-floor metric meets the tolerance too."""
    wl = wls.resnet50_cifar100()
    run_and_check(wl, cols=windows(wl, width=1024, n_random=1024, boundaries=6), steps=8, shuffle=True, plain=True)


def test_shuffle_reconcile_refusals():
    dev = torch.device("cuda")
    W, N = 4, 4 * 1024
    g = torch.randn(W, N, device=dev) * 1e-3
    with CPDPState(W, N, **HYPER) as st:
        st.init_params(torch.zeros(N, device=dev))
        st.set_reconcile_shuffle(True)
        with pytest.raises(cpdp.CPDPError) as e:
            st.set_reconcile_staging(2)
        assert e.value.status == cpdp.CPDP_ESTATE
        for setup in (lambda: st.set_method("localsgd"), lambda: st.set_state_reconcile(True)):
            setup()
            with pytest.raises(cpdp.CPDPError) as e:
                st.reconcile(g)
            assert e.value.status == cpdp.CPDP_ESTATE and "shuffle" in str(e.value)
            st.set_method("cpdp")
            st.set_state_reconcile(False)
        with pytest.raises(cpdp.CPDPError) as e:
            st.reconcile(g.to(torch.bfloat16))
        assert e.value.status == cpdp.CPDP_ESTATE
        st.reconcile(g)
        st.set_reconcile_shuffle(False)
        st.set_reconcile_staging(2)
        with pytest.raises(cpdp.CPDPError) as e:
            st.set_reconcile_shuffle(True)
        assert e.value.status == cpdp.CPDP_ESTATE
    with CPDPState(2, 66, **HYPER) as st:
        with pytest.raises(cpdp.CPDPError) as e:
            st.set_reconcile_shuffle(True)
        assert e.value.status == cpdp.CPDP_EINVAL and "multiple of 4" in str(e.value)


@pytest.mark.parametrize("W,N,option,want", [
    (8, 4 * 300, None, "reconcile_vec4_kernel"),
    (2, 4 * 300, None, "reconcile_onepass_kernel"),
    (1, 4 * 300, None, "reconcile_onepass_kernel"),
    (8, 4 * 300 + 3, None, "reconcile_scalar_kernel"),
    (8, 4 * 300, "shuffle", "reconcile_shuffle_kernel"),
    (8, 4 * 300, "staging", "reconcile_tma_kernel"),
])
def test_reconcile_kernel_names_the_kernel_that_ran(W, N, option, want):
    """cpdp_reconcile_kernel reports the kernel the dispatch chose, for the
    default vectorised shape, the one-pass kernel (SGD with float32 gradients
    at W = 1 and 2), the scalar kernel (N not a multiple of 4) and the two
    opt-in mappings."""
    dev = torch.device("cuda")
    with CPDPState(W, N, **HYPER) as st:
        st.init_params(torch.zeros(N, device=dev))
        if option == "shuffle":
            st.set_reconcile_shuffle(True)
        elif option == "staging":
            st.set_reconcile_staging(3)
        assert st.reconcile_kernel() == ""
        st.step(torch.zeros(W, N, device=dev), 1, 2)  # a local step leaves it unset
        assert st.reconcile_kernel() == ""
        st.step(torch.zeros(W, N, device=dev), 2, 2)
        torch.cuda.synchronize()
        assert st.reconcile_kernel() == want
