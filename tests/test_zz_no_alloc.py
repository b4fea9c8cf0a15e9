"""cpdp_step_host_noalloc: the host-fed step for callers that cannot allocate
device memory of their own (their device memory belongs to another allocator,
or their step loop must not call cudaMalloc). It stages the gradients in an
area built into the library instead of the buffers cpdp_bind_staging needs.

Its results are compared with the existing host-fed step, cpdp_step_host with
bound staging buffers, on the same inputs over two calls in a row: a local
step, then a reconcile. This file is collected last, so a run that stops at
the first failure has run every other test before it."""
import numpy as np
import pytest
import torch

from paper_2607_21224_gb300 import cpdp
from paper_2607_21224_gb300.pipeline import HostGradientPipeline
from paper_2607_21224_gb300.state import CPDPState, grad_dtype_code
from parity import TOL, scaled_error

pytestmark = pytest.mark.gpu


def _arrays(st):
    return [st.params, st.mom, st.anchor, st.slow_v]


@pytest.mark.parametrize("N,gdt", [(4 * 2501, torch.float32), (4 * 2501, torch.bfloat16), (1027, torch.float32)])
def test_noalloc_host_step_matches_staged_host_step(N, gdt):
    W, K, T = 4, 2, 2
    dev = torch.device("cuda")
    gen = torch.Generator(device="cpu").manual_seed(7)
    theta0 = (torch.randn(N, generator=gen) * 0.05).to(dev)
    host = [(torch.randn(W, N, generator=gen) * 1e-3).to(gdt).pin_memory() for _ in range(T)]
    code = grad_dtype_code(host[0])
    hyper = dict(lr=0.1, momentum=0.9, weight_decay=5e-4, K=K, beta=0.5)
    with CPDPState(W, N, **hyper) as staged, CPDPState(W, N, **hyper) as noalloc:
        staged.init_params(theta0)
        noalloc.init_params(theta0)
        feed = HostGradientPipeline(staged, dtype=gdt)
        stream = torch.cuda.current_stream().cuda_stream
        for t in range(1, T + 1):  # t = 1: local step; t = 2 = K: reconcile
            want = feed.step(host[t - 1], t, T)
            got = cpdp.cpdp_step_host_noalloc(noalloc.ctx, host[t - 1], code, t, T, stream)
            assert got == want == (t == K)
            torch.cuda.synchronize()
            tid = np.zeros(N, dtype=np.int64)
            for x, y in zip(_arrays(noalloc), _arrays(staged)):
                assert scaled_error(x.double().cpu().numpy(), y.double().cpu().numpy(), tid) <= TOL
                assert torch.equal(x.view(torch.int32), y.view(torch.int32))


def test_noalloc_rejects_a_step_beyond_the_built_in_area():
    W = 8
    N = cpdp.CPDP_NOALLOC_STAGING_BYTES // (4 * W) + 4  # float32 gradients one vector past the limit
    with CPDPState(W, N, lr=0.1, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5) as st:
        st.init_params(torch.zeros(N, device="cuda"))
        host = torch.ones(W, N).pin_memory()
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_step_host_noalloc(st.ctx, host, cpdp.CPDP_F32, 1, 2)
        assert e.value.status == cpdp.CPDP_EINVAL and "built-in staging area" in str(e.value)
        torch.cuda.synchronize()
        assert int(torch.count_nonzero(st.params)) == 0  # nothing was launched
        # the same step in bfloat16 takes half the bytes and fits; the pinned
        # tensor stays referenced until the copy has run
        host_bf16 = host.to(torch.bfloat16).pin_memory()
        assert not cpdp.cpdp_step_host_noalloc(st.ctx, host_bf16, cpdp.CPDP_BF16, 1, 2)
        torch.cuda.synchronize()
        assert int(torch.count_nonzero(st.params)) > 0


def _captured_node_count(call, stream) -> tuple[int, Exception | None]:
    """Run `call` while `stream` is captured into a CUDA graph (driver API,
    relaxed mode); return the captured graph's node count and what `call`
    raised."""
    import ctypes
    cu = ctypes.CDLL("libcuda.so.1")
    h = ctypes.c_void_p(stream.cuda_stream)
    assert cu.cuStreamBeginCapture_v2(h, 2) == 0  # CU_STREAM_CAPTURE_MODE_RELAXED
    raised = None
    try:
        call()
    except Exception as e:  # noqa: BLE001 - returned to the caller
        raised = e
    graph = ctypes.c_void_p()
    assert cu.cuStreamEndCapture(h, ctypes.byref(graph)) == 0
    n = ctypes.c_size_t(0)
    assert cu.cuGraphGetNodes(graph, None, ctypes.byref(n)) == 0
    assert cu.cuGraphDestroy(graph) == 0
    return n.value, raised


def test_noalloc_adamw_refused_under_capture_before_any_copy():
    """AdamW's step cannot be replayed from a graph (its bias correction moves
    with the step count), so the call is refused under capture; the refusal
    comes before the gradients' copy, and the captured graph stays empty."""
    W, N = 2, 4 * 1024
    host = (torch.randn(W, N) * 1e-3).pin_memory()
    with CPDPState(W, N, lr=1e-3, momentum=0.0, weight_decay=0.05, K=2, beta=0.5) as st:
        st.set_adamw()
        st.init_params(torch.randn(N, device="cuda") * 0.05)
        side = torch.cuda.Stream()
        assert not cpdp.cpdp_step_host_noalloc(st.ctx, host, cpdp.CPDP_F32, 1, 2, side.cuda_stream)
        side.synchronize()
        before = st.params.clone()
        nodes, raised = _captured_node_count(
            lambda: cpdp.cpdp_step_host_noalloc(st.ctx, host, cpdp.CPDP_F32, 2, 2, side.cuda_stream), side)
        assert isinstance(raised, cpdp.CPDPError) and raised.status == cpdp.CPDP_ESTATE, raised
        assert nodes == 0
        assert st.optimizer_step == 1 and torch.equal(st.params, before)
        assert cpdp.cpdp_step_host_noalloc(st.ctx, host, cpdp.CPDP_F32, 2, 2, side.cuda_stream)  # eager: runs
        side.synchronize()
        assert st.optimizer_step == 2
