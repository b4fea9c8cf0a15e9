"""CUDA path (through the C ABI) against the fp64 oracle on the same seeded
inputs, element by element, after every step. Tolerance: the scaled error of
tests/parity.py must stay within 1e-5 for float32 and bfloat16 gradients alike
(the oracle receives the exact bfloat16 values, so the bf16 variant carries no
extra error; the looser 1e-2 bound allowed for it is not needed), and all W
replicas must be bit-identical after every reconcile."""
import json

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21224_gb300 import cpdp
from paper_2607_21224_gb300 import workloads as wls
from paper_2607_21224_gb300.state import CPDPState
from parity import TOL, Pair, oracle_hyper, run_and_check, windows
from oracle_pins import GOLDEN_CASES, load_golden

pytestmark = pytest.mark.gpu


def flat(name, N, W, K, T, grad_dtype="f32", tensors=1, **kw):
    return wls.Workload(name, W=W, tensors=tuple(wls.flat_tensors(N, tensors, 0.05)), K=K, T=T,
                        grad_dtype=grad_dtype, **kw)


# ---------------------------------------------------------------------------
# worked examples: dyadic values, so the GPU must match bit for bit
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", GOLDEN_CASES)
@pytest.mark.parametrize("pad", [0, 1])
def test_golden_bit_exact(name, pad):
    """The hand-derived examples of tests/golden, on the vector path (N=4) and,
    with one extra zero column (N=5), on the scalar path."""
    c = load_golden(name)
    W, N = c["W"], c["N"] + pad
    dev = torch.device("cuda")
    theta0 = torch.tensor(c["theta0"] + [0.0] * pad, dtype=torch.float32, device=dev)
    with CPDPState(W, N, None, lr=c["lr"], momentum=c["momentum"], weight_decay=c["weight_decay"],
                   K=c["K"], beta=c["beta"], alpha=c["alpha"], device=dev) as st:
        st.init_params(theta0)
        for g, want in zip(c["grads"], c["after"]):
            grads = torch.tensor([row + [0.0] * pad for row in g], dtype=torch.float32, device=dev)
            assert st.step(grads, want["t"], c["T"]) == want["sync"]
            torch.cuda.synchronize()
            for key, attr in (("theta", "params"), ("buf", "mom"), ("theta_ref", "anchor"), ("v", "slow_v")):
                got = getattr(st, attr).cpu()
                exp = torch.tensor(want[key], dtype=torch.float32)
                if pad:
                    got = got[..., :-1]
                assert torch.equal(got, exp), (name, want["t"], key, got.tolist(), exp.tolist())


# ---------------------------------------------------------------------------
# the small configuration, every element
# ---------------------------------------------------------------------------
def test_tiny_full_epoch():
    worst = run_and_check(wls.tiny(), plain=True)
    assert all(v <= TOL for v in worst.values()) and worst.plain <= TOL


@pytest.mark.parametrize("N", [1, 2, 3, 4, 5, 7, 8, 13, 37, 1000, 1001, 1027, 4096 + 3])
@pytest.mark.parametrize("W", [1, 3, 8])
def test_ragged_sizes(N, W):
    """Odd and tiny N (scalar reconcile path and the local step's ragged tail),
    with T=5, K=2 so the epoch-end rule adds a reconcile at t=5."""
    run_and_check(flat(f"ragged_{N}_{W}", N, W, K=2, T=5))


@pytest.mark.parametrize("W", [2, 5, 8, 9, 16, 32])
def test_multi_tile_vector_path(W):
    """Vector path over many blocks with a partial last block (N/4 not a
    multiple of the block size), W not a multiple of the 8-row chunk for 5 and 9."""
    run_and_check(flat(f"tiles_W{W}", 4 * (256 * 37 + 11), W, K=3, T=7, tensors=5))


def test_bf16_gradients_small():
    run_and_check(flat("bf16_small", 40_000, 8, K=4, T=8, grad_dtype="bf16", tensors=3))


def test_heavy_tail_small():
    run_and_check(flat("heavy_small", 50_000, 16, K=2, T=6, heavy_tail_p=0.01, beta=0.7))


@pytest.mark.parametrize("kw", [
    dict(K=1, beta=0.0, alpha=1.0),             # synchronous DDP
    dict(K=1, beta=0.9, alpha=1.0),             # SlowMo every step
    dict(K=3, beta=0.3, alpha=0.5),             # alpha != 1
    dict(K=2, beta=0.5, momentum=0.0, weight_decay=0.0),  # plain SGD (eq. 5 literally)
    dict(K=100, beta=0.5),                      # only the epoch-end reconcile
])
def test_hyperparameter_corners(kw):
    run_and_check(flat("corner", 12_345 * 4, 4, T=6, **kw))


# ---------------------------------------------------------------------------
# the paper-shaped configurations at full size (windowed oracle)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["resnet50_cifar100", "vit_s16_cifar100", "resnet50_tinyimagenet"])
def test_full_size_configs(name):
    wl = wls.get(name)
    run_and_check(wl, cols=windows(wl), plain=True)


@pytest.mark.parametrize("N,W,K", wls.sweep_points(), ids=lambda v: str(v))
def test_sweep_points(N, W, K):
    """Every roofline-sweep point (76), the largest (N=2^28, W=16: 51.5 GB of
    state and gradients) included, through one full K-cycle and the next local
    step in the launch shapes the benchmark times; every column checked up to
    2^23 elements per array, sampled columns beyond."""
    wl = wls.sweep_point(N, W, K)
    cols = None if W * N <= (1 << 23) else windows(wl, width=512, n_random=1024, boundaries=0)
    run_and_check(wl, cols=cols, steps=min(wl.T, K + 1), plain=True)


# ---------------------------------------------------------------------------
# semantics that are unique and checkable directly
# ---------------------------------------------------------------------------
def test_momentum_buffers_stay_per_worker():
    """Sec. 4.2: the reconcile does not touch the buffers' locality: after a
    reconcile with distinct gradients the buffers still differ across workers."""
    wl = flat("buffers", 4096, 4, K=2, T=2)
    pair = Pair(wl)
    try:
        pair.step(1)
        pair.step(2)
        torch.cuda.synchronize()
        b = pair.gpu.mom
        assert not torch.equal(b[0], b[1])
        assert pair.replicas_identical()
    finally:
        pair.close()


def test_worker_permutation_bitwise():
    """Eqs. 2 and 7 do not depend on worker order. Small-integer data keep every
    float32 sum exact, so permuted workers give bit-identical anchors and v."""
    W, N = 4, 64
    dev = torch.device("cuda")
    gen = torch.Generator().manual_seed(5)
    theta0 = torch.randint(-8, 8, (N,), generator=gen).float().to(dev)
    grads = [torch.randint(-4, 5, (W, N), generator=gen).float().to(dev) for _ in range(4)]
    perm = torch.tensor([3, 1, 0, 2], device=dev)
    hp = dict(lr=0.5, momentum=0.5, weight_decay=0.0, K=2, beta=0.5, alpha=1.0)
    with CPDPState(W, N, **hp) as a, CPDPState(W, N, **hp) as b:
        a.init_params(theta0)
        b.init_params(theta0)
        for t, g in enumerate(grads, start=1):
            a.step(g, t, 4)
            b.step(g[perm].contiguous(), t, 4)
        torch.cuda.synchronize()
        assert torch.equal(a.anchor, b.anchor) and torch.equal(a.slow_v, b.slow_v)
        assert torch.equal(a.mom[perm], b.mom) and torch.equal(a.params[perm], b.params)


def test_checkpoint_resume_bit_identical(tmp_path):
    """All state is in caller-owned buffers: 2 steps + save + fresh context +
    load + 2 steps equals 4 steps straight, bit for bit."""
    wl = wls.tiny()
    dev = torch.device("cuda")
    theta0 = wls.make_theta0(wl, 42, dev)
    grads = [wls.make_grads(wl, t, 42, dev) for t in range(1, 5)]
    with CPDPState(wl.W, wl.N, wl.offsets, **wl.hyper()) as a:
        a.init_params(theta0)
        for t in range(1, 5):
            a.step(grads[t - 1], t, wl.T)
        straight = [x.clone() for x in (a.params, a.mom, a.anchor, a.slow_v)]
    with CPDPState(wl.W, wl.N, wl.offsets, **wl.hyper()) as b:
        b.init_params(theta0)
        for t in range(1, 3):
            b.step(grads[t - 1], t, wl.T)
        torch.save({k: getattr(b, k).cpu() for k in ("params", "mom", "anchor", "slow_v")}, tmp_path / "ck.pt")
    ck = torch.load(tmp_path / "ck.pt")
    with CPDPState(wl.W, wl.N, wl.offsets, **wl.hyper()) as c:
        for k, v in ck.items():
            getattr(c, k).copy_(v)
        for t in range(3, 5):
            c.step(grads[t - 1], t, wl.T)
        torch.cuda.synchronize()
        for x, y in zip(straight, (c.params, c.mom, c.anchor, c.slow_v)):
            assert torch.equal(x, y)


def test_pinned_host_gradients_match_device():
    """Gradients may live in page-locked host memory (read over the
    CPU-GPU link); the result is bit-identical to device-resident gradients."""
    wl = flat("pinned", 4 * 5000, 4, K=2, T=4)
    dev = torch.device("cuda")
    theta0 = wls.make_theta0(wl, 1, dev)
    with CPDPState(wl.W, wl.N, **wl.hyper()) as a, CPDPState(wl.W, wl.N, **wl.hyper()) as b:
        a.init_params(theta0)
        b.init_params(theta0)
        for t in range(1, 5):
            g = wls.make_grads(wl, t, 1, dev)
            a.step(g, t, wl.T)
            b.step(g.cpu().pin_memory(), t, wl.T)
            torch.cuda.synchronize()
        assert torch.equal(a.params, b.params) and torch.equal(a.mom, b.mom)
        assert torch.equal(a.anchor, b.anchor) and torch.equal(a.slow_v, b.slow_v)


def test_non_default_stream():
    wl = flat("stream", 4 * 3000, 3, K=2, T=4)
    s = torch.cuda.Stream()
    pair = Pair(wl)
    try:
        with torch.cuda.stream(s):
            for t in range(1, 5):
                pair.step(t)
            s.synchronize()
            errs = pair.errors()
        assert all(e <= TOL for e in errs.values()), errs
    finally:
        pair.close()


def test_set_lr_changes_following_steps():
    """cpdp_set_lr (a caller-driven schedule) takes effect at the next step:
    matches the oracle run with the same per-step learning rates."""
    wl = flat("lr_sched", 4 * 2000, 2, K=2, T=4)
    lrs = [0.1, 0.05, 0.025, 0.2]
    pair = Pair(wl)
    try:
        for t in range(1, 5):
            pair.gpu.set_lr(lrs[t - 1])
            pair.hp.lr = float(np.float32(lrs[t - 1]))
            pair.step(t)
        errs = pair.errors()
        assert all(e <= TOL for e in errs.values()), errs
    finally:
        pair.close()


# ---------------------------------------------------------------------------
# argument errors that need device memory to provoke (host-side checks)
# ---------------------------------------------------------------------------
def test_gradient_argument_errors():
    W, N = 2, 64
    with CPDPState(W, N, lr=0.1, momentum=0.9, weight_decay=0.0, K=2, beta=0.5) as st:
        st.init_params(torch.zeros(N, device="cuda"))
        g = torch.zeros(W * N + 4, device="cuda")
        with pytest.raises(cpdp.CPDPError) as e:          # misaligned by 4 bytes
            cpdp.cpdp_local_step(st.ctx, g.data_ptr() + 4, cpdp.CPDP_F32, 0)
        assert e.value.status == cpdp.CPDP_EALIGN
        with pytest.raises(cpdp.CPDPError) as e:          # overlaps the replicas
            cpdp.cpdp_reconcile(st.ctx, st.params.data_ptr(), cpdp.CPDP_F32, 0)
        assert e.value.status == cpdp.CPDP_EINVAL
        pageable = torch.zeros(W * N)                     # plain host memory
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_local_step(st.ctx, pageable.data_ptr(), cpdp.CPDP_F32, 0)
        assert e.value.status == cpdp.CPDP_EINVAL
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_local_step(st.ctx, g.data_ptr(), 7, 0)
        assert e.value.status == cpdp.CPDP_EINVAL
        # the context is still usable after rejected calls
        st.local_step(torch.zeros(W, N, device="cuda"))
        torch.cuda.synchronize()


def test_init_params_rejects_pageable_host_theta0():
    with CPDPState(2, 64, lr=0.1, momentum=0.9, weight_decay=0.0, K=2, beta=0.5) as st:
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_init_params(st.ctx, torch.zeros(64), 0)
        assert e.value.status == cpdp.CPDP_EINVAL
        st.init_params(torch.zeros(64).pin_memory())  # page-locked host memory is readable
        torch.cuda.synchronize()
        assert torch.equal(st.params.cpu(), torch.zeros(2, 64))


def test_bind_rejects_host_memory():
    ctx = cpdp.cpdp_create(2, 64, None, 0.1, 0.9, 0.0, 2, 0.5, 1.0)
    try:
        host = [torch.zeros(2 * 64), torch.zeros(2 * 64), torch.zeros(64), torch.zeros(64)]
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_bind(ctx, *host)
        assert e.value.status == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


# ---------------------------------------------------------------------------
# training-protocol schedule and CUDA-graph replay
# ---------------------------------------------------------------------------
def test_protocol_schedule_parity():
    """Three epochs through cpdp_step_at (warmup epoch at K = 1, cosine LR)
    against the oracle driven by its own schedule functions, every step."""
    wl = flat("protocol", 4 * 2500, 3, K=2, T=5, tensors=2)
    E, We, base, lo = 3, 1, 0.1, 1e-3
    pair = Pair(wl)
    pair.gpu.set_schedule(wl.T, E, We, base, lo)
    b32, l32 = float(np.float32(base)), float(np.float32(lo))
    try:
        for e in range(E):
            for t in range(1, wl.T + 1):
                s = e * wl.T + t - 1
                pair.hp.lr = float(np.float32(pair.orc.scheduled_lr(b32, l32, We * wl.T, E * wl.T, s)))
                step = e * wl.T + t
                wls.make_grads(wl, step, pair.seed, pair.device, out=pair.grads)
                synced = pair.gpu.step_at(pair.grads, e, t)
                g = pair._host(pair.grads)
                want = pair.orc.is_sync_step_at(e, t, wl.K, wl.T, We)
                assert synced == want
                (pair.orc.reconcile if want else pair.orc.local_step)(pair.ost, g, pair.hp)
                errs = pair.errors()
                assert all(x <= TOL for x in errs.values()), (e, t, errs)
                if synced:
                    assert pair.replicas_identical()
    finally:
        pair.close()


def test_cuda_graph_k_cycle_replay():
    """A K-cycle captured into a CUDA graph and replayed equals eager execution
    bit for bit (the entry points are capture-safe once a gradient buffer's
    pointer has been checked by an eager call)."""
    wl = flat("graph", 4 * 4096, 4, K=4, T=4)
    dev = torch.device("cuda")
    theta0 = wls.make_theta0(wl, 3, dev)
    grads = [wls.make_grads(wl, t, 3, dev) for t in range(1, 5)]
    with CPDPState(wl.W, wl.N, **wl.hyper()) as eager, CPDPState(wl.W, wl.N, **wl.hyper()) as graphed:
        eager.init_params(theta0)
        graphed.init_params(theta0)
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):  # eager warm-up call per buffer (pointer checks happen here)
            for k in range(4):
                graphed.local_step(grads[k])
        torch.cuda.current_stream().wait_stream(s)
        for k in range(4):
            eager.local_step(grads[k])
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for k in range(4):
                graphed.step(grads[k], k + 1, 4)
        for _ in range(3):
            for k in range(4):
                eager.step(grads[k], k + 1, 4)
            g.replay()
        torch.cuda.synchronize()
        for a, b in ((eager.params, graphed.params), (eager.mom, graphed.mom),
                     (eager.anchor, graphed.anchor), (eager.slow_v, graphed.slow_v)):
            assert torch.equal(a, b)


@pytest.mark.parametrize("method,opt,state_sync,gd,N", [
    ("cpdp", "sgd", False, "f32", 4 * (256 * 9 + 5)), ("cpdp", "adamw", True, "bf16", 4 * 3001),
    ("localsgd", "sgd", False, "bf16", 4 * 2000), ("ddp", "adamw", False, "f32", 4 * 1500),
    ("cpdp", "sgd", False, "f32", 1027),
])
def test_pdl_bit_identical_to_plain_launches(method, opt, state_sync, gd, N):
    """Programmatic dependent launches (the default) and plain stream-ordered
    launches give bit-identical state through two K-cycles."""
    W, K, T = 5, 3, 6
    dev = torch.device("cuda")
    gdt = torch.float32 if gd == "f32" else torch.bfloat16
    gen = torch.Generator(device=dev).manual_seed(11)
    theta0 = torch.randn(N, device=dev, generator=gen) * 0.05
    grads = [(torch.randn(W, N, device=dev, generator=gen) * 1e-3).to(gdt) for _ in range(T)]
    out = []
    for pdl in (True, False):
        lr = 1e-3 if opt == "adamw" else 0.1
        with CPDPState(W, N, lr=lr, momentum=0.9, weight_decay=5e-4, K=K, beta=0.5) as st:
            if opt == "adamw":
                st.set_adamw()
            st.set_pdl(pdl)
            st.set_method(method)
            st.set_state_reconcile(state_sync)
            st.init_params(theta0)
            for t in range(1, T + 1):
                st.step(grads[t - 1], t, T)
            torch.cuda.synchronize()
            arrays = [st.params, st.mom, st.anchor, st.slow_v] + ([st.exp_avg_sq] if opt == "adamw" else [])
            out.append([x.clone() for x in arrays])
    for a, b in zip(*out):
        assert torch.equal(a.view(torch.int32), b.view(torch.int32))


def _refused_under_capture(call):
    """Run `call` while torch captures a CUDA graph on its side stream; return
    the CPDPError status it raised."""
    g = torch.cuda.CUDAGraph()
    marker = torch.zeros(1, device="cuda")
    with pytest.raises(cpdp.CPDPError) as e:
        with torch.cuda.graph(g):
            marker.add_(1)  # one captured node, so the graph is not empty
            call()
    torch.cuda.synchronize()
    return e.value.status


def test_graph_capture_refused_where_replay_would_be_stale():
    """AdamW steps, schedule-driven steps and host-fed steps return
    CPDP_ESTATE under stream capture and launch nothing; the context keeps
    working eagerly afterwards, with its counters unchanged by the refusals."""
    from paper_2607_21224_gb300.pipeline import HostGradientPipeline
    dev = torch.device("cuda")
    N, W = 4 * 1024, 2
    g = torch.randn(W, N, device=dev) * 1e-3
    theta0 = torch.randn(N, device=dev) * 0.05
    with CPDPState(W, N, lr=1e-3, momentum=0.0, weight_decay=0.05, K=2, beta=0.5) as st:
        st.set_adamw()
        st.init_params(theta0)
        st.local_step(g)  # eager call: the gradient pointer is checked here
        before = st.params.clone()
        assert _refused_under_capture(lambda: st.local_step(g)) == cpdp.CPDP_ESTATE
        assert _refused_under_capture(lambda: st.reconcile(g)) == cpdp.CPDP_ESTATE
        assert "CUDA graph" in cpdp.cpdp_last_error(st.ctx)
        assert st.optimizer_step == 1 and torch.equal(st.params, before)
        st.local_step(g)
        assert st.optimizer_step == 2
    with CPDPState(W, N, lr=0.1, momentum=0.9, weight_decay=5e-4, K=2, beta=0.5) as st:
        st.init_params(theta0)
        st.set_schedule(2, 2, 0, 0.1, 0.0)
        st.step_at(g, 0, 1)
        assert _refused_under_capture(lambda: st.step_at(g, 0, 2)) == cpdp.CPDP_ESTATE
        assert st.counts() == (0, 0)
        feed = HostGradientPipeline(st)
        host = g.cpu().pin_memory()
        assert _refused_under_capture(lambda: feed.step(host, 1, 2)) == cpdp.CPDP_ESTATE
        assert st.step_at(g, 0, 2) and st.counts() == (1, 1)  # eager steps still run


# ---------------------------------------------------------------------------
# the paper's baselines on the same kernels (Sec. 5.4)
# ---------------------------------------------------------------------------
from oracle_pins import METHOD_CASES  # noqa: E402


@pytest.mark.parametrize("name", METHOD_CASES)
def test_method_golden_bit_exact(name):
    c = load_golden(name)
    dev = torch.device("cuda")
    with CPDPState(c["W"], c["N"], None, lr=c["lr"], momentum=c["momentum"], weight_decay=c["weight_decay"],
                   K=c["K"], beta=c["beta"], alpha=c["alpha"], device=dev) as st:
        st.init_params(torch.tensor(c["theta0"], dtype=torch.float32, device=dev))
        st.set_method(c["method"])
        for g, want in zip(c["grads"], c["after"]):
            assert st.step(torch.tensor(g, dtype=torch.float32, device=dev), want["t"], c["T"]) == want["sync"]
            torch.cuda.synchronize()
            for key, attr in (("theta", "params"), ("buf", "mom"), ("theta_ref", "anchor"), ("v", "slow_v")):
                got = getattr(st, attr).cpu()
                assert torch.equal(got, torch.tensor(want[key], dtype=torch.float32)), (name, want["t"], key)


@pytest.mark.parametrize("W", [1, 2, 3, 4, 5, 6])
@pytest.mark.parametrize("method,state_sync", [("cpdp", False), ("cpdp", True), ("localsgd", False),
                                               ("localsgd", True), ("ddp", False)])
@pytest.mark.parametrize("opt", ["sgd", "adamw"])
@pytest.mark.parametrize("gd", ["f32", "bf16"])
def test_few_workers_every_variant(W, method, state_sync, opt, gd):
    """One to six workers, where the reconcile's shape depends on the worker
    count (one round trip, or chunks of 1-4 rows, per variant): every method,
    optimizer, state reconciliation and gradient type against the oracle, over
    several blocks with a partial last one."""
    N = 4 * (256 * 5 + 3)
    if opt == "adamw":
        wl = flat(f"few_{W}", N, W, K=2, T=5, grad_dtype=gd, tensors=2, lr=5e-4, weight_decay=0.05, momentum=0.0,
                  optimizer="adamw")
    else:
        wl = flat(f"few_{W}", N, W, K=2, T=5, grad_dtype=gd, tensors=2)
    run_and_check(wl, method=method, state_sync=state_sync)


@pytest.mark.parametrize("W", [7, 8, 12, 16])
@pytest.mark.parametrize("method", ["cpdp", "ddp"])
@pytest.mark.parametrize("opt,gd", [("sgd", "bf16"), ("adamw", "bf16"), ("adamw", "f32")])
def test_many_workers_gradient_chunks(W, method, opt, gd):
    """From 7 workers on, CPDP and DDP reconcile SGD with bf16 gradients and
    AdamW with gradient-row chunks of 8 (bf16) or 4 (float32) held as raw
    words and 4- or 3-row state chunks, the first loaded with the gradients:
    full and partial chunks of both kinds, over several blocks with a partial
    last one, against the oracle."""
    N = 4 * (256 * 5 + 3)
    if opt == "adamw":
        wl = flat(f"gc_{W}", N, W, K=2, T=5, grad_dtype=gd, tensors=2, lr=5e-4, weight_decay=0.05, momentum=0.0,
                  optimizer="adamw")
    else:
        wl = flat(f"gc_{W}", N, W, K=2, T=5, grad_dtype=gd, tensors=2)
    run_and_check(wl, method=method)


@pytest.mark.parametrize("method", ["localsgd", "ddp"])
@pytest.mark.parametrize("N,W,gd", [(4 * (256 * 21 + 5), 8, "f32"), (1027, 3, "f32"), (40_000, 5, "bf16"),
                                    (4 * 3000, 16, "f32")])
def test_method_parity(method, N, W, gd):
    run_and_check(flat(f"{method}_{N}_{W}", N, W, K=3, T=7, grad_dtype=gd, tensors=2), method=method)


@pytest.mark.parametrize("method", ["cpdp", "localsgd", "ddp"])
def test_method_full_size_resnet50(method):
    wl = wls.get("resnet50_cifar100")
    run_and_check(wl, cols=windows(wl, width=1024, n_random=1024, boundaries=6), steps=8, method=method)


def test_table2_counts_per_epoch():
    """Table 2: per epoch of T steps, DDP launches T gradient means and no
    parameter means; LocalSGD none and ceil(T/K); CPDP ceil(T/K) of each."""
    T, K = 11, 4
    wl = flat("counts", 4 * 1024, 4, K=K, T=T)
    dev = torch.device("cuda")
    g = wls.make_grads(wl, 1, 1, dev)
    want = {"ddp": (T, 0), "localsgd": (0, -(-T // K)), "cpdp": (-(-T // K), -(-T // K))}
    for method, counts in want.items():
        with CPDPState(wl.W, wl.N, **wl.hyper()) as st:
            st.init_params(wls.make_theta0(wl, 1, dev))
            st.set_method(method)
            syncs = sum(st.step(g, t, T) for t in range(1, T + 1))
            torch.cuda.synchronize()
            assert st.counts() == counts, (method, st.counts())
            assert syncs == (T if method == "ddp" else -(-T // K))


# ---------------------------------------------------------------------------
# AdamW as the workers' optimizer (the paper's ViT-S runs)
# ---------------------------------------------------------------------------
def adamw(name, N, W, K, T, grad_dtype="f32", tensors=2, **kw):
    return flat(name, N, W, K, T, grad_dtype=grad_dtype, tensors=tensors, lr=5e-4, weight_decay=0.05,
                momentum=0.0, optimizer="adamw", **kw)


@pytest.mark.parametrize("method", ["cpdp", "localsgd", "ddp"])
@pytest.mark.parametrize("N,W,gd", [(4 * (256 * 13 + 7), 8, "f32"), (4 * 5000, 5, "bf16"), (1027, 3, "f32"),
                                    (999, 4, "bf16"), (4 * 3001, 7, "bf16"), (4 * 2003, 12, "f32"),
                                    (4 * 1501, 16, "bf16")])
def test_adamw_parity(method, N, W, gd):
    run_and_check(adamw(f"adamw_{method}_{N}", N, W, K=3, T=7, grad_dtype=gd), method=method)


def test_adamw_full_size_vit():
    """The paper's ViT-S optimizer at full size. The floors raise some
    denominators (governed_frac > 0), but every element also meets the
    tolerance without any floor, so at this configuration they decide
    nothing."""
    wl = wls.get("vit_s16_cifar100_adamw")
    worst = run_and_check(wl, cols=windows(wl), plain=True)
    assert 0.0 < worst.governed_frac <= 1.0 and worst.max_floor_ratio > 1.0
    assert worst.plain <= TOL, worst.plain


@pytest.mark.parametrize("method,state_sync", [("localsgd", False), ("ddp", False), ("cpdp", True),
                                               ("localsgd", True)])
def test_adamw_full_size_vit_variants(method, state_sync):
    """The paper's ViT-S optimizer at full size with the baselines' sync steps
    and with state reconciliation, in the launch shapes the benchmark times."""
    wl = wls.get("vit_s16_cifar100_adamw")
    run_and_check(wl, cols=windows(wl, width=1024, n_random=1024, boundaries=6), steps=8, method=method,
                  state_sync=state_sync, plain=True)


@pytest.mark.parametrize("opt,method", [("adamw", "cpdp"), ("sgd", "cpdp"), ("sgd", "ddp")])
def test_largest_size_reconcile_with_64_bit_offsets(opt, method):
    """The largest state this suite builds: W = 8 workers with bf16 gradients
    over N = 2^30 + 4 parameters (AdamW: 112 GB of state; SGD: 77 GB; 17 GB of
    gradients). Here W * N / 4 plus the grid's threads exceeds 2^31, so the
    reconcile's gradient-chunk shape runs with 64-bit offsets instead of the
    32-bit ones it uses below that size. Sampled columns (head, tail, random)
    against the oracle through a local step, a reconcile and the epoch-end
    reconcile; replicas bit-identical on the whole arrays after each CPDP
    reconcile."""
    N = (1 << 30) + 4
    if opt == "adamw":
        wl = adamw("largest", N, 8, K=2, T=3, grad_dtype="bf16", tensors=1)
    else:
        wl = flat("largest", N, 8, K=2, T=3, grad_dtype="bf16", tensors=1)
    assert (wl.W + 1) * N > 1 << 33
    run_and_check(wl, method=method, cols=windows(wl, width=512, n_random=2048, boundaries=0))


def test_adamw_optimizer_step_and_resume(tmp_path):
    """The shared AdamW step count advances once per step and restarts at
    cpdp_init_params; resuming from saved buffers plus the step count is
    bit-identical to running straight through."""
    wl = adamw("adamw_resume", 4 * 3000, 4, K=2, T=4)
    dev = torch.device("cuda")
    theta0 = wls.make_theta0(wl, 5, dev)
    grads = [wls.make_grads(wl, t, 5, dev) for t in range(1, 5)]

    def fresh():
        st = CPDPState(wl.W, wl.N, **wl.hyper())
        st.set_adamw()
        return st

    with fresh() as a:
        a.init_params(theta0)
        assert a.optimizer_step == 0
        for t in range(1, 5):
            a.step(grads[t - 1], t, wl.T)
        assert a.optimizer_step == 4
        straight = [x.clone() for x in (a.params, a.mom, a.exp_avg_sq, a.anchor, a.slow_v)]
    with fresh() as b:
        b.init_params(theta0)
        for t in range(1, 3):
            b.step(grads[t - 1], t, wl.T)
        saved = {k: getattr(b, k).cpu() for k in ("params", "mom", "exp_avg_sq", "anchor", "slow_v")}
        saved_step = b.optimizer_step
    with fresh() as c:
        for k, v in saved.items():
            getattr(c, k).copy_(v)
        c.optimizer_step = saved_step
        for t in range(3, 5):
            c.step(grads[t - 1], t, wl.T)
        torch.cuda.synchronize()
        for x, y in zip(straight, (c.params, c.mom, c.exp_avg_sq, c.anchor, c.slow_v)):
            assert torch.equal(x, y)


def test_set_adamw_argument_errors():
    with CPDPState(2, 64, lr=1e-3, momentum=0.0, weight_decay=0.0, K=2, beta=0.5) as st:
        sq = torch.zeros(2 * 64 + 4, device="cuda")
        for bad in ((1.0, 0.999, 1e-8), (0.9, -0.1, 1e-8), (0.9, 0.999, -1.0)):
            with pytest.raises(cpdp.CPDPError) as e:
                cpdp.cpdp_set_adamw(st.ctx, *bad, sq)
            assert e.value.status == cpdp.CPDP_EINVAL
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_set_adamw(st.ctx, 0.9, 0.999, 1e-8, sq.data_ptr() + 4)
        assert e.value.status == cpdp.CPDP_EALIGN
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_set_adamw(st.ctx, 0.9, 0.999, 1e-8, st.mom)
        assert e.value.status == cpdp.CPDP_EINVAL
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_set_adamw(st.ctx, 0.9, 0.999, 1e-8, torch.zeros(2 * 64))
        assert e.value.status == cpdp.CPDP_EINVAL


# ---------------------------------------------------------------------------
# optimizer-state reconciliation (the variant the paper names)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("method", ["cpdp", "localsgd"])
@pytest.mark.parametrize("opt", ["sgd", "adamw"])
@pytest.mark.parametrize("N,W,gd", [(4 * (256 * 11 + 3), 8, "f32"), (4 * 3001, 5, "bf16"), (1031, 3, "f32")])
def test_state_reconcile_parity(method, opt, N, W, gd):
    mk = adamw if opt == "adamw" else flat
    kw = {} if opt == "adamw" else dict(tensors=2)
    run_and_check(mk(f"ss_{method}_{opt}_{N}", N, W, K=3, T=7, grad_dtype=gd, **kw), method=method,
                  state_sync=True)


def test_state_reconcile_full_size_resnet50():
    wl = wls.get("resnet50_cifar100")
    run_and_check(wl, cols=windows(wl, width=1024, n_random=1024, boundaries=6), steps=8, state_sync=True)


# ---------------------------------------------------------------------------
# host-fed gradients (end-to-end use through HostGradientPipeline)
# ---------------------------------------------------------------------------
def test_host_gradient_pipeline_matches_device_resident():
    """Gradients copied from pinned host memory on a copy stream, overlapped
    with earlier steps, give bit-identical state to device-resident gradients."""
    from paper_2607_21224_gb300.pipeline import HostGradientPipeline
    wl = flat("pipe", 4 * 20_000, 4, K=3, T=6)
    dev = torch.device("cuda")
    theta0 = wls.make_theta0(wl, 9, dev)
    host = [wls.make_grads(wl, t, 9, "cpu").pin_memory() for t in range(1, 7)]
    with CPDPState(wl.W, wl.N, **wl.hyper()) as a, CPDPState(wl.W, wl.N, **wl.hyper()) as b:
        a.init_params(theta0)
        b.init_params(theta0)
        feed = HostGradientPipeline(b)
        s = torch.cuda.Stream()
        for t in range(1, 7):
            a.step(host[t - 1].to(dev), t, wl.T)
            feed.step(host[t - 1], t, wl.T, stream=s)
        torch.cuda.synchronize()
        for x, y in ((a.params, b.params), (a.mom, b.mom), (a.anchor, b.anchor), (a.slow_v, b.slow_v)):
            assert torch.equal(x, y)
        with pytest.raises(ValueError):
            feed.step(host[0].clone(), 1, wl.T)  # not pinned


@pytest.mark.parametrize("W", [64, 257, 1024, 4096])
def test_many_workers(W):
    """Worker counts up to the ABI's limit (4096), vector and scalar paths."""
    for N in (4 * 33, 37):
        run_and_check(flat(f"many_{W}_{N}", N, W, K=2, T=3))


def test_two_contexts_on_two_host_threads():
    """Distinct contexts are independent: two host threads, each driving its own
    CPDPState on its own stream, give the same results as running them one
    after the other."""
    import threading
    wls_ = [flat(f"thr{i}", 4 * 8000, 3 + i, K=2, T=4) for i in range(2)]
    dev = torch.device("cuda")
    inputs = [(wls.make_theta0(wl, 20 + i, dev), [wls.make_grads(wl, t, 20 + i, dev) for t in range(1, 5)])
              for i, wl in enumerate(wls_)]

    def run(i, out):
        wl = wls_[i]
        theta0, grads = inputs[i]
        s = torch.cuda.Stream()
        with torch.cuda.stream(s):
            with CPDPState(wl.W, wl.N, **wl.hyper()) as st:
                st.init_params(theta0, stream=s)
                for t in range(1, 5):
                    st.step(grads[t - 1], t, wl.T, stream=s)
                s.synchronize()
                out[i] = [x.clone() for x in (st.params, st.mom, st.anchor, st.slow_v)]

    seq, par = {}, {}
    for i in range(2):
        run(i, seq)
    threads = [threading.Thread(target=run, args=(i, par)) for i in range(2)]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    for i in range(2):
        assert all(torch.equal(a, b) for a, b in zip(seq[i], par[i]))


def test_host_staging_argument_errors_and_protocol():
    """cpdp_bind_staging's checks, and cpdp_step_host_at against device-fed
    cpdp_step_at over a short protocol (bit-identical)."""
    from paper_2607_21224_gb300.pipeline import HostGradientPipeline
    wl = flat("staging", 4 * 3000, 3, K=2, T=4)
    dev = torch.device("cuda")
    with CPDPState(wl.W, wl.N, **wl.hyper()) as st:
        small = torch.empty(16, device=dev)
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_bind_staging(st.ctx, small, small.data_ptr() + 1 << 10, 64)
        assert e.value.status in (cpdp.CPDP_EINVAL, cpdp.CPDP_EALIGN)
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_bind_staging(st.ctx, st.params, torch.empty(wl.W * wl.N, device=dev), 4 * wl.W * wl.N)
        assert e.value.status == cpdp.CPDP_EINVAL
        with pytest.raises(cpdp.CPDPError) as e:
            cpdp.cpdp_bind_staging(st.ctx, torch.empty(wl.W * wl.N), torch.empty(wl.W * wl.N), 4 * wl.W * wl.N)
        assert e.value.status == cpdp.CPDP_EINVAL
    theta0 = wls.make_theta0(wl, 4, dev)
    host = [wls.make_grads(wl, t, 4, "cpu").pin_memory() for t in range(1, 9)]
    with CPDPState(wl.W, wl.N, **wl.hyper()) as a, CPDPState(wl.W, wl.N, **wl.hyper()) as b:
        for x in (a, b):
            x.init_params(theta0)
            x.set_schedule(wl.T, 2, 1, 0.1, 0.001)
        feed = HostGradientPipeline(b)
        for e in range(2):
            for t in range(1, wl.T + 1):
                g = host[e * wl.T + t - 1]
                assert a.step_at(g.to(dev), e, t) == feed.step_at(g, e, t)
        torch.cuda.synchronize()
        for x, y in ((a.params, b.params), (a.mom, b.mom), (a.anchor, b.anchor), (a.slow_v, b.slow_v)):
            assert torch.equal(x, y)
