"""Pins that tie the fp64 oracle to what the paper and the mathematics fix.

Each pin takes an ``oracle.OracleLib`` and raises AssertionError when the
library disagrees with something other than itself:

* hand-derived worked examples (``tests/golden/*.json``; dyadic values, so the
  expected results are exact),
* library routines the method reduces to in a special case
  (``torch.optim.SGD`` in float64, ``numpy.mean``),
* closed forms (the SlowMo velocity under a constant drift is a geometric
  series; the number of synchronizations per epoch is ceil(T/K), Table 2),
* invariants (worker permutation, identical replicas).

The same pins run against deliberately broken copies of the oracle
(tests/test_oracle_mutants.py) to show that each plausible mistake is caught.
"""
from __future__ import annotations

import json
import math
from pathlib import Path

import numpy as np
import torch

from oracle import Hyper, OracleLib

GOLDEN_DIR = Path(__file__).resolve().parent / "golden"
GOLDEN_CASES = sorted(p.name for p in GOLDEN_DIR.glob("case_*.json"))
METHOD_CASES = sorted(p.name for p in GOLDEN_DIR.glob("method_*.json"))


def load_golden(name: str) -> dict:
    return json.loads((GOLDEN_DIR / name).read_text())


def _hyper(case: dict) -> Hyper:
    return Hyper(lr=case["lr"], momentum=case["momentum"], weight_decay=case["weight_decay"],
                 K=case["K"], beta=case["beta"], alpha=case["alpha"])


def _torch_sgd(theta0, grads, lr, mu, wd):
    """Textbook momentum SGD (torch.optim.SGD, float64, CPU) over a gradient sequence."""
    p = torch.nn.Parameter(torch.tensor(np.asarray(theta0), dtype=torch.float64))
    opt = torch.optim.SGD([p], lr=lr, momentum=mu, weight_decay=wd, foreach=False)
    for g in grads:
        p.grad = torch.tensor(np.asarray(g), dtype=torch.float64)
        opt.step()
    buf = opt.state[p].get("momentum_buffer")
    buf = np.zeros_like(np.asarray(theta0)) if buf is None else buf.numpy().copy()
    return p.detach().numpy().copy(), buf


# --------------------------------------------------------------------------
# hand-derived worked examples (exact)
# --------------------------------------------------------------------------
def pin_golden(lib: OracleLib, name: str) -> None:
    case = load_golden(name)
    hp = _hyper(case)
    st = lib.init(case["W"], np.array(case["theta0"], dtype=np.float64))
    for t, (g, want) in enumerate(zip(case["grads"], case["after"]), start=1):
        assert want["t"] == t
        synced = lib.step(st, np.array(g, dtype=np.float64), hp, t, case["T"], case.get("method", "cpdp"))
        assert synced == want["sync"], f"{name} t={t}: sync flag {synced} != {want['sync']}"
        for key in ("theta", "buf", "theta_ref", "v"):
            got = getattr(st, key)
            exp = np.array(want[key], dtype=np.float64)
            assert np.array_equal(got, exp), f"{name} t={t} {key}: {got.tolist()} != {exp.tolist()}"


# --------------------------------------------------------------------------
# special cases that reduce to library routines
# --------------------------------------------------------------------------
def pin_sgd_single_worker(lib: OracleLib) -> None:
    """W=1, K=1, beta=0, alpha=1: CPDP is plain momentum SGD (K=1 is synchronous
    training, Sec. 3.1; beta=0 removes the SlowMo term)."""
    rng = np.random.default_rng(7)
    N, T = 33, 12
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, 1, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=1, beta=0.0, alpha=1.0)
    st = lib.init(1, theta0)
    for t in range(1, T + 1):
        assert lib.step(st, grads[t - 1], hp, t, T)
    ref_theta, ref_buf = _torch_sgd(theta0, grads[:, 0, :], hp.lr, hp.momentum, hp.weight_decay)
    np.testing.assert_allclose(st.theta[0], ref_theta, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(st.buf[0], ref_buf, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(st.theta_ref, ref_theta, rtol=1e-12, atol=1e-15)


def pin_ddp_k1(lib: OracleLib) -> None:
    """K=1, beta=0, alpha=1 with W=3 distinct gradients: every replica follows
    synchronous data-parallel SGD on the mean gradient (eqs. 2-3, Sec. 3.1)."""
    rng = np.random.default_rng(11)
    W, N, T = 3, 17, 6
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.05, momentum=0.9, weight_decay=5e-4, K=1, beta=0.0, alpha=1.0)
    st = lib.init(W, theta0)
    for t in range(1, T + 1):
        lib.step(st, grads[t - 1], hp, t, T)
    mean_grads = np.mean(grads, axis=1)
    ref_theta, ref_buf = _torch_sgd(theta0, mean_grads, hp.lr, hp.momentum, hp.weight_decay)
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], ref_theta, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], ref_buf, rtol=1e-12, atol=1e-15)


def pin_local_steps_independent(lib: OracleLib) -> None:
    """Local phase (eq. 5): each worker is an independent SGD optimizer on its own
    gradients; nothing crosses workers."""
    rng = np.random.default_rng(3)
    W, N, T = 3, 21, 5
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=100, beta=0.5, alpha=1.0)
    st = lib.init(W, theta0)
    for t in range(T):
        lib.local_step(st, grads[t], hp)
    for i in range(W):
        ref_theta, ref_buf = _torch_sgd(theta0, grads[:, i, :], hp.lr, hp.momentum, hp.weight_decay)
        np.testing.assert_allclose(st.theta[i], ref_theta, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], ref_buf, rtol=1e-12, atol=1e-15)
    # the anchor and the velocity are untouched by local steps
    assert np.array_equal(st.theta_ref, theta0)
    assert np.array_equal(st.v, np.zeros(N))


def pin_optimizer_state_stays_local(lib: OracleLib) -> None:
    """Sync step with beta=0, alpha=1 (Sec. 3.2 stages one and two, Sec. 4.2):
    each worker's own SGD optimizer applies the mean gradient; the momentum
    buffers are not averaged; the parameters become the mean of the post-step
    replicas. Driven here by W independent torch.optim.SGD instances and numpy.mean."""
    rng = np.random.default_rng(5)
    W, N, K, T = 3, 19, 2, 4
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=K, beta=0.0, alpha=1.0)
    st = lib.init(W, theta0)
    for t in range(1, T + 1):
        lib.step(st, grads[t - 1], hp, t, T)

    params = [torch.nn.Parameter(torch.tensor(theta0, dtype=torch.float64)) for _ in range(W)]
    opts = [torch.optim.SGD([p], lr=hp.lr, momentum=hp.momentum, weight_decay=hp.weight_decay,
                            foreach=False) for p in params]
    for t in range(1, T + 1):
        sync = (t % K == 0) or (t == T)
        gbar = np.mean(grads[t - 1], axis=0)
        for i in range(W):
            params[i].grad = torch.tensor(gbar if sync else grads[t - 1, i])
            opts[i].step()
        if sync:
            avg = np.mean(np.stack([p.detach().numpy() for p in params]), axis=0)
            with torch.no_grad():
                for p in params:
                    p.copy_(torch.tensor(avg))
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], params[i].detach().numpy(), rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], opts[i].state[params[i]]["momentum_buffer"].numpy(),
                                   rtol=1e-12, atol=1e-15)
    # buffers really differ across workers (they were not reconciled)
    assert not np.allclose(st.buf[0], st.buf[1])


def pin_mean_gradient(lib: OracleLib) -> None:
    """A single reconcile from the initial state with mu=0, wd=0, lr=1, beta=0,
    alpha=1 moves every replica by minus the mean gradient (eqs. 2, 6, 7, 10)."""
    rng = np.random.default_rng(9)
    W, N = 3, 13
    theta0 = rng.normal(0.0, 1.0, N)
    g = rng.normal(0.0, 1.0, (W, N))
    st = lib.init(W, theta0)
    lib.reconcile(st, g, Hyper(lr=1.0, momentum=0.0, weight_decay=0.0, K=1, beta=0.0, alpha=1.0))
    expect = theta0 - np.mean(g, axis=0)
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], expect, rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(st.v, expect - theta0, rtol=1e-12, atol=1e-15)


# --------------------------------------------------------------------------
# closed forms
# --------------------------------------------------------------------------
def pin_slowmo_geometric(lib: OracleLib) -> None:
    """Constant drift: with mu=0, wd=0, K=1 and the same gradient g on every
    worker at every step, each reconcile sees delta = -lr*g. Eqs. 8-10 then give
    v_n = delta (1 - beta^n) / (1 - beta) and
    theta_ref_n = theta0 + alpha * delta / (1-beta) * (n - beta (1 - beta^n) / (1 - beta))."""
    rng = np.random.default_rng(13)
    W, N, n = 2, 11, 7
    lr, beta, alpha = 0.1, 0.7, 0.8
    theta0 = rng.normal(0.0, 1.0, N)
    g = rng.normal(0.0, 1.0, N)
    hp = Hyper(lr=lr, momentum=0.0, weight_decay=0.0, K=1, beta=beta, alpha=alpha)
    st = lib.init(W, theta0)
    for t in range(1, n + 1):
        assert lib.step(st, np.stack([g] * W), hp, t, n)
        delta = -lr * g
        v_t = delta * (1 - beta ** t) / (1 - beta)
        ref_t = theta0 + alpha * delta / (1 - beta) * (t - beta * (1 - beta ** t) / (1 - beta))
        np.testing.assert_allclose(st.v, v_t, rtol=1e-10, atol=1e-13)
        np.testing.assert_allclose(st.theta_ref, ref_t, rtol=1e-10, atol=1e-13)
        for i in range(W):
            np.testing.assert_allclose(st.theta[i], ref_t, rtol=1e-10, atol=1e-13)


def pin_schedule_counts(lib: OracleLib) -> None:
    """Eq. 4 plus the epoch-end rule: syncs fall at t = K, 2K, ... and at t = T,
    ceil(T/K) of them per epoch (Table 2, CPDP row)."""
    for T in range(1, 41):
        for K in range(1, 13):
            syncs = [t for t in range(1, T + 1) if lib.is_sync_step(t, K, T)]
            assert len(syncs) == math.ceil(T / K), (T, K, syncs)
            assert syncs[-1] == T, (T, K, syncs)
            assert set(range(K, T + 1, K)) <= set(syncs), (T, K, syncs)
    # K = 1 synchronizes every step (synchronous DDP, Sec. 3.1)
    assert all(lib.is_sync_step(t, 1, 9) for t in range(1, 10))


# --------------------------------------------------------------------------
# invariants
# --------------------------------------------------------------------------
def pin_permutation_invariance(lib: OracleLib) -> None:
    """The means of eqs. 2 and 7 do not depend on worker order: permuting the
    workers permutes theta and buf rows and leaves theta_ref and v unchanged.
    Small-integer data keep every sum exact, so the check is bit-exact."""
    rng = np.random.default_rng(17)
    W, N, K, T = 4, 8, 3, 7
    theta0 = rng.integers(-8, 8, N).astype(np.float64)
    grads = rng.integers(-4, 5, (T, W, N)).astype(np.float64)
    hp = Hyper(lr=0.5, momentum=0.5, weight_decay=0.0, K=K, beta=0.5, alpha=1.0)
    perm = np.array([2, 0, 3, 1])
    a, b = lib.init(W, theta0), lib.init(W, theta0)
    for t in range(1, T + 1):
        lib.step(a, grads[t - 1], hp, t, T)
        lib.step(b, grads[t - 1][perm], hp, t, T)
        assert np.array_equal(a.theta[perm], b.theta)
        assert np.array_equal(a.buf[perm], b.buf)
        assert np.array_equal(a.theta_ref, b.theta_ref)
        assert np.array_equal(a.v, b.v)


def pin_identical_replicas_identity(lib: OracleLib) -> None:
    """Reconciling identical replicas with nothing to apply (zero gradients, zero
    weight decay, empty momentum, v = 0) returns them unchanged (Sec. 3.3: the
    average of identical models is that model, delta = 0, v stays 0)."""
    rng = np.random.default_rng(19)
    W, N = 4, 10
    theta0 = rng.normal(0.0, 1.0, N)
    st = lib.init(W, theta0)
    lib.reconcile(st, np.zeros((W, N)), Hyper(lr=0.1, momentum=0.9, weight_decay=0.0,
                                              K=1, beta=0.5, alpha=1.0))
    for i in range(W):
        assert np.array_equal(st.theta[i], theta0)
    assert np.array_equal(st.theta_ref, theta0)
    assert np.array_equal(st.v, np.zeros(N))


def pin_identical_gradients_match_local(lib: OracleLib) -> None:
    """With the same gradient on every worker and identical replicas, the
    reconcile's synced step is the local step (gbar = g); with v = 0, beta
    arbitrary and alpha = 1, theta_new = theta_ref + (theta' - theta_ref) = theta'
    up to one rounding."""
    rng = np.random.default_rng(23)
    W, N = 4, 15
    theta0 = rng.normal(0.0, 0.05, N)
    g = rng.normal(0.0, 1e-2, N)
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=1, beta=0.9, alpha=1.0)
    a, b = lib.init(W, theta0), lib.init(W, theta0)
    lib.reconcile(a, np.stack([g] * W), hp)
    lib.local_step(b, np.stack([g] * W), hp)
    np.testing.assert_allclose(a.theta, b.theta, rtol=1e-14, atol=1e-16)
    assert np.array_equal(a.buf, b.buf)


# --------------------------------------------------------------------------
# training-protocol schedule (Sec. 4.3, Sec. 5.4)
# --------------------------------------------------------------------------
def pin_lr_schedule_vs_torch(lib: OracleLib) -> None:
    """Linear warmup, then cosine annealing: the warmup part equals
    torch.optim.lr_scheduler.LinearLR(start_factor=1/Sw, total_iters=Sw-1) and the
    rest equals CosineAnnealingLR(T_max=S-Sw, eta_min), each driven on its own."""
    for base, lo, Sw, S in ((0.4, 0.0, 35, 140), (0.1, 1e-3, 8, 50), (5e-4, 0.0, 2, 9)):
        opt = torch.optim.SGD([torch.nn.Parameter(torch.zeros(1))], lr=base)
        sch = torch.optim.lr_scheduler.LinearLR(opt, start_factor=1.0 / Sw, end_factor=1.0, total_iters=Sw - 1)
        for s in range(Sw):
            want = opt.param_groups[0]["lr"]
            got = lib.scheduled_lr(base, lo, Sw, S, s)
            assert math.isclose(got, want, rel_tol=1e-12, abs_tol=1e-18), (s, got, want)
            opt.step()
            sch.step()
        opt = torch.optim.SGD([torch.nn.Parameter(torch.zeros(1))], lr=base)
        sch = torch.optim.lr_scheduler.CosineAnnealingLR(opt, T_max=S - Sw, eta_min=lo)
        for s in range(Sw, S):
            want = opt.param_groups[0]["lr"]
            got = lib.scheduled_lr(base, lo, Sw, S, s)
            assert math.isclose(got, want, rel_tol=1e-9, abs_tol=1e-15), (s, got, want)
            opt.step()
            sch.step()


def pin_lr_schedule_closed_forms(lib: OracleLib) -> None:
    """Values fixed by the shape alone: base/Sw at the first step, base at the
    end of warmup and at the start of the decay, (base+min)/2 halfway, and
    min + (base-min)(1+sqrt(2)/2)/2 a quarter of the way (a linear decay would
    give 3/4 there); strictly above min until the end; no warmup when Sw = 0."""
    base, lo, Sw, S = 0.4, 0.01, 20, 420
    assert math.isclose(lib.scheduled_lr(base, lo, Sw, S, 0), base / Sw, rel_tol=1e-15)
    assert math.isclose(lib.scheduled_lr(base, lo, Sw, S, Sw - 1), base, rel_tol=1e-15)
    assert math.isclose(lib.scheduled_lr(base, lo, Sw, S, Sw), base, rel_tol=1e-15)
    assert math.isclose(lib.scheduled_lr(base, lo, Sw, S, Sw + 200), (base + lo) / 2, rel_tol=1e-14)
    q = lo + (base - lo) * (1 + math.sqrt(2) / 2) / 2
    assert math.isclose(lib.scheduled_lr(base, lo, Sw, S, Sw + 100), q, rel_tol=1e-14)
    decay = [lib.scheduled_lr(base, lo, Sw, S, s) for s in range(Sw, S)]
    assert all(a > b for a, b in zip(decay, decay[1:])) and decay[-1] > lo
    assert math.isclose(lib.scheduled_lr(base, lo, 0, 10, 0), base, rel_tol=1e-15)


def pin_warmup_sync_counts(lib: OracleLib) -> None:
    """During the warmup epochs every step synchronizes (K = 1, Sec. 4.3);
    afterwards eq. 4 with the epoch-end rule gives ceil(T/K) syncs per epoch
    (Table 2 counts apply to post-warmup epochs)."""
    for T, K, E, We in ((7, 2, 5, 2), (16, 4, 3, 1), (5, 8, 4, 0)):
        total = 0
        for e in range(E):
            n = sum(lib.is_sync_step_at(e, t, K, T, We) for t in range(1, T + 1))
            assert n == (T if e < We else math.ceil(T / K)), (T, K, e, We, n)
            total += n
        assert total == We * T + (E - We) * math.ceil(T / K)


# --------------------------------------------------------------------------
# the paper's baselines (Sec. 5.4): DDP and LocalSGD
# --------------------------------------------------------------------------
def pin_ddp_vs_torch(lib: OracleLib) -> None:
    """DDP: every worker follows torch.optim.SGD on the mean gradient (eqs. 2-3)."""
    rng = np.random.default_rng(29)
    W, N, T = 3, 23, 6
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=4, beta=0.5, alpha=1.0)
    st = lib.init(W, theta0)
    for t in range(1, T + 1):
        assert lib.step(st, grads[t - 1], hp, t, T, "ddp")
    ref_theta, ref_buf = _torch_sgd(theta0, np.mean(grads, axis=1), hp.lr, hp.momentum, hp.weight_decay)
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], ref_theta, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], ref_buf, rtol=1e-12, atol=1e-15)
    assert np.array_equal(st.theta_ref, theta0) and not st.v.any()


def pin_localsgd_vs_torch(lib: OracleLib) -> None:
    """LocalSGD: W independent torch.optim.SGD optimizers on their own
    gradients; at t = K, 2K, ... and at the epoch's end, numpy.mean of the
    parameters is written back to all; buffers stay per worker."""
    rng = np.random.default_rng(31)
    W, N, K, T = 3, 19, 2, 5
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=K, beta=0.5, alpha=1.0)
    st = lib.init(W, theta0)
    for t in range(1, T + 1):
        lib.step(st, grads[t - 1], hp, t, T, "localsgd")
    params = [torch.nn.Parameter(torch.tensor(theta0, dtype=torch.float64)) for _ in range(W)]
    opts = [torch.optim.SGD([p], lr=hp.lr, momentum=hp.momentum, weight_decay=hp.weight_decay,
                            foreach=False) for p in params]
    for t in range(1, T + 1):
        for i in range(W):
            params[i].grad = torch.tensor(grads[t - 1, i])
            opts[i].step()
        if t % K == 0 or t == T:
            avg = np.mean(np.stack([p.detach().numpy() for p in params]), axis=0)
            with torch.no_grad():
                for p in params:
                    p.copy_(torch.tensor(avg))
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], params[i].detach().numpy(), rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], opts[i].state[params[i]]["momentum_buffer"].numpy(),
                                   rtol=1e-12, atol=1e-15)
    assert np.array_equal(st.theta_ref, theta0) and not st.v.any()


def pin_first_sync_linearity(lib: OracleLib) -> None:
    """With a momentum-SGD step (linear in the gradient), averaging after
    per-worker steps equals stepping with the mean gradient: at the first
    synchronization (v = 0, alpha = 1) CPDP and LocalSGD give the same
    parameters; their momentum buffers differ (mean vs own gradient)."""
    rng = np.random.default_rng(37)
    W, N, K = 4, 29, 3
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (K, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=K, beta=0.7, alpha=1.0)
    a, b = lib.init(W, theta0), lib.init(W, theta0)
    for t in range(1, K + 1):
        lib.step(a, grads[t - 1], hp, t, K, "cpdp")
        lib.step(b, grads[t - 1], hp, t, K, "localsgd")
    np.testing.assert_allclose(a.theta, b.theta, rtol=1e-12, atol=1e-15)
    assert not np.allclose(a.buf, b.buf)


def pin_ddp_equals_cpdp_k1_beta0(lib: OracleLib) -> None:
    """DDP is CPDP with K = 1, beta = 0, alpha = 1 (Sec. 3.1): same parameters up
    to rounding (CPDP averages identical replicas and adds a zero velocity) and
    identical momentum buffers."""
    rng = np.random.default_rng(41)
    W, N, T = 3, 17, 5
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=1, beta=0.0, alpha=1.0)
    a, b = lib.init(W, theta0), lib.init(W, theta0)
    for t in range(1, T + 1):
        lib.step(a, grads[t - 1], hp, t, T, "cpdp")
        lib.step(b, grads[t - 1], hp, t, T, "ddp")
    np.testing.assert_allclose(a.theta, b.theta, rtol=1e-13, atol=1e-16)
    np.testing.assert_allclose(a.buf, b.buf, rtol=1e-13, atol=1e-16)


# --------------------------------------------------------------------------
# AdamW as the workers' optimizer (the paper's ViT-S runs, Sec. 5.2, Table 3)
# --------------------------------------------------------------------------
def _torch_adamw(theta0, grads, lr, wd, betas=(0.9, 0.999), eps=1e-8):
    p = torch.nn.Parameter(torch.tensor(np.asarray(theta0), dtype=torch.float64))
    opt = torch.optim.AdamW([p], lr=lr, betas=betas, eps=eps, weight_decay=wd, foreach=False)
    for g in grads:
        p.grad = torch.tensor(np.asarray(g), dtype=torch.float64)
        opt.step()
    st = opt.state[p]
    return p.detach().numpy().copy(), st["exp_avg"].numpy().copy(), st["exp_avg_sq"].numpy().copy()


def pin_adamw_single_worker_vs_torch(lib: OracleLib) -> None:
    """W = 1, K = 1, beta = 0, alpha = 1: the AdamW variant is torch.optim.AdamW."""
    from oracle import AdamWOracle
    rng = np.random.default_rng(43)
    N, T = 31, 10
    theta0 = rng.normal(0.0, 0.02, N)
    grads = rng.normal(0.0, 1e-3, (T, 1, N))
    hp = Hyper(lr=5e-4, momentum=0.0, weight_decay=0.05, K=1, beta=0.0, alpha=1.0)
    ad = AdamWOracle(lib)
    st = ad.init(1, theta0)
    for t in range(1, T + 1):
        assert ad.step(st, grads[t - 1], hp, t, T)
    th, m, sq = _torch_adamw(theta0, grads[:, 0, :], hp.lr, hp.weight_decay)
    np.testing.assert_allclose(st.theta[0], th, rtol=1e-10, atol=1e-15)
    np.testing.assert_allclose(st.buf[0], m, rtol=1e-12, atol=1e-18)
    np.testing.assert_allclose(st.sq[0], sq, rtol=1e-12, atol=1e-20)


def pin_adamw_ddp_k1(lib: OracleLib) -> None:
    """K = 1, beta = 0, alpha = 1, W = 3: every replica follows torch AdamW on the
    mean gradient, with identical per-worker moments."""
    from oracle import AdamWOracle
    rng = np.random.default_rng(47)
    W, N, T = 3, 21, 6
    theta0 = rng.normal(0.0, 0.02, N)
    grads = rng.normal(0.0, 1e-3, (T, W, N))
    hp = Hyper(lr=5e-4, momentum=0.0, weight_decay=0.05, K=1, beta=0.0, alpha=1.0)
    ad = AdamWOracle(lib, 0.8, 0.99, 1e-7)
    st = ad.init(W, theta0)
    for t in range(1, T + 1):
        ad.step(st, grads[t - 1], hp, t, T)
    th, m, sq = _torch_adamw(theta0, np.mean(grads, axis=1), hp.lr, hp.weight_decay, (0.8, 0.99), 1e-7)
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], th, rtol=1e-10, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], m, rtol=1e-12, atol=1e-18)
        np.testing.assert_allclose(st.sq[i], sq, rtol=1e-12, atol=1e-20)


def pin_adamw_state_stays_local(lib: OracleLib) -> None:
    """Local AdamW steps on own gradients, a sync step with the mean gradient
    through each worker's own moments, then the parameter mean (beta = 0): W
    torch AdamW instances and numpy.mean give the same parameters and moments."""
    from oracle import AdamWOracle
    rng = np.random.default_rng(53)
    W, N, K, T = 3, 17, 2, 4
    theta0 = rng.normal(0.0, 0.02, N)
    grads = rng.normal(0.0, 1e-3, (T, W, N))
    hp = Hyper(lr=5e-4, momentum=0.0, weight_decay=0.05, K=K, beta=0.0, alpha=1.0)
    ad = AdamWOracle(lib)
    st = ad.init(W, theta0)
    for t in range(1, T + 1):
        ad.step(st, grads[t - 1], hp, t, T)
    params = [torch.nn.Parameter(torch.tensor(theta0, dtype=torch.float64)) for _ in range(W)]
    opts = [torch.optim.AdamW([p], lr=hp.lr, weight_decay=hp.weight_decay, foreach=False) for p in params]
    for t in range(1, T + 1):
        sync = (t % K == 0) or (t == T)
        gbar = np.mean(grads[t - 1], axis=0)
        for i in range(W):
            params[i].grad = torch.tensor(gbar if sync else grads[t - 1, i])
            opts[i].step()
        if sync:
            avg = np.mean(np.stack([p.detach().numpy() for p in params]), axis=0)
            with torch.no_grad():
                for p in params:
                    p.copy_(torch.tensor(avg))
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], params[i].detach().numpy(), rtol=1e-10, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], opts[i].state[params[i]]["exp_avg"].numpy(), rtol=1e-12, atol=1e-18)
        np.testing.assert_allclose(st.sq[i], opts[i].state[params[i]]["exp_avg_sq"].numpy(), rtol=1e-12, atol=1e-20)
    assert not np.allclose(st.buf[0], st.buf[1])


def pin_adamw_slowmo_geometric(lib: OracleLib) -> None:
    """Constant gradient g on every worker, K = 1, no weight decay: bias
    correction makes m_hat = g and s_hat = g^2 at every step, so each reconcile
    sees delta = -lr g / (|g| + eps) and v follows the geometric closed form."""
    from oracle import AdamWOracle
    rng = np.random.default_rng(59)
    W, N, n = 2, 9, 6
    lr, beta, alpha, eps = 1e-3, 0.6, 0.9, 1e-8
    theta0 = rng.normal(0.0, 1.0, N)
    g = rng.normal(0.0, 1e-2, N)
    ad = AdamWOracle(lib, eps=eps)
    hp = Hyper(lr=lr, momentum=0.0, weight_decay=0.0, K=1, beta=beta, alpha=alpha)
    st = ad.init(W, theta0)
    delta = -lr * g / (np.abs(g) + eps)
    for t in range(1, n + 1):
        ad.step(st, np.stack([g] * W), hp, t, n)
        v_t = delta * (1 - beta ** t) / (1 - beta)
        ref_t = theta0 + alpha * delta / (1 - beta) * (t - beta * (1 - beta ** t) / (1 - beta))
        np.testing.assert_allclose(st.v, v_t, rtol=1e-9, atol=1e-15)
        np.testing.assert_allclose(st.theta_ref, ref_t, rtol=1e-9, atol=1e-15)


def pin_adamw_baselines_vs_torch(lib: OracleLib) -> None:
    """AdamW under the paper's baselines: DDP = torch AdamW on the mean gradient
    for every worker; LocalSGD = W torch AdamW instances on their own gradients
    with numpy.mean of the parameters written back at t = K, 2K, ... and T."""
    from oracle import AdamWOracle
    rng = np.random.default_rng(61)
    W, N, K, T = 3, 13, 2, 5
    theta0 = rng.normal(0.0, 0.02, N)
    grads = rng.normal(0.0, 1e-3, (T, W, N))
    hp = Hyper(lr=5e-4, momentum=0.0, weight_decay=0.05, K=K, beta=0.5, alpha=1.0)
    ad = AdamWOracle(lib)
    ddp = ad.init(W, theta0)
    for t in range(1, T + 1):
        ad.step(ddp, grads[t - 1], hp, t, T, "ddp")
    th, m, sq = _torch_adamw(theta0, np.mean(grads, axis=1), hp.lr, hp.weight_decay)
    for i in range(W):
        np.testing.assert_allclose(ddp.theta[i], th, rtol=1e-10, atol=1e-15)
        np.testing.assert_allclose(ddp.sq[i], sq, rtol=1e-12, atol=1e-20)
    loc = ad.init(W, theta0)
    for t in range(1, T + 1):
        ad.step(loc, grads[t - 1], hp, t, T, "localsgd")
    params = [torch.nn.Parameter(torch.tensor(theta0, dtype=torch.float64)) for _ in range(W)]
    opts = [torch.optim.AdamW([p], lr=hp.lr, weight_decay=hp.weight_decay, foreach=False) for p in params]
    for t in range(1, T + 1):
        for i in range(W):
            params[i].grad = torch.tensor(grads[t - 1, i])
            opts[i].step()
        if t % K == 0 or t == T:
            avg = np.mean(np.stack([p.detach().numpy() for p in params]), axis=0)
            with torch.no_grad():
                for p in params:
                    p.copy_(torch.tensor(avg))
    for i in range(W):
        np.testing.assert_allclose(loc.theta[i], params[i].detach().numpy(), rtol=1e-10, atol=1e-15)
        np.testing.assert_allclose(loc.buf[i], opts[i].state[params[i]]["exp_avg"].numpy(), rtol=1e-12, atol=1e-18)


# --------------------------------------------------------------------------
# optimizer-state reconciliation (Sec. 4.2's named variant)
# --------------------------------------------------------------------------
def pin_state_sync_vs_torch(lib: OracleLib) -> None:
    """CPDP with optimizer-state reconciliation, driven independently: W torch
    SGD optimizers step on their own gradients between syncs; at a sync each
    steps with the mean gradient, then numpy.mean of the parameters (beta = 0,
    alpha = 1) and of the momentum buffers is written back to every worker."""
    rng = np.random.default_rng(67)
    W, N, K, T = 3, 15, 2, 5
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=K, beta=0.0, alpha=1.0)
    st = lib.init(W, theta0)
    for t in range(1, T + 1):
        lib.step(st, grads[t - 1], hp, t, T, "cpdp", state_sync=True)
    params = [torch.nn.Parameter(torch.tensor(theta0, dtype=torch.float64)) for _ in range(W)]
    opts = [torch.optim.SGD([p], lr=hp.lr, momentum=hp.momentum, weight_decay=hp.weight_decay,
                            foreach=False) for p in params]
    for t in range(1, T + 1):
        sync = (t % K == 0) or (t == T)
        gbar = np.mean(grads[t - 1], axis=0)
        for i in range(W):
            params[i].grad = torch.tensor(gbar if sync else grads[t - 1, i])
            opts[i].step()
        if sync:
            avg = np.mean(np.stack([p.detach().numpy() for p in params]), axis=0)
            bufs = [opts[i].state[params[i]]["momentum_buffer"] for i in range(W)]
            bavg = np.mean(np.stack([b.numpy() for b in bufs]), axis=0)
            with torch.no_grad():
                for p, b in zip(params, bufs):
                    p.copy_(torch.tensor(avg))
                    b.copy_(torch.tensor(bavg))
    for i in range(W):
        np.testing.assert_allclose(st.theta[i], params[i].detach().numpy(), rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(st.buf[i], opts[i].state[params[i]]["momentum_buffer"].numpy(),
                                   rtol=1e-12, atol=1e-15)


def pin_state_sync_makes_cpdp_k1_ddp(lib: OracleLib) -> None:
    """With K = 1 the buffers enter every sync identical, so state averaging is
    neutral: CPDP (beta = 0, alpha = 1) with and without it, and DDP, agree."""
    rng = np.random.default_rng(71)
    W, N, T = 4, 11, 5
    theta0 = rng.normal(0.0, 0.05, N)
    grads = rng.normal(0.0, 1e-2, (T, W, N))
    hp = Hyper(lr=0.1, momentum=0.9, weight_decay=5e-4, K=1, beta=0.0, alpha=1.0)
    a, b, c = lib.init(W, theta0), lib.init(W, theta0), lib.init(W, theta0)
    for t in range(1, T + 1):
        lib.step(a, grads[t - 1], hp, t, T, "cpdp", state_sync=True)
        lib.step(b, grads[t - 1], hp, t, T, "cpdp")
        lib.step(c, grads[t - 1], hp, t, T, "ddp")
    np.testing.assert_allclose(a.buf, b.buf, rtol=1e-14, atol=1e-17)
    np.testing.assert_allclose(a.buf, c.buf, rtol=1e-14, atol=1e-17)
    np.testing.assert_allclose(a.theta, c.theta, rtol=1e-13, atol=1e-16)


def pin_average_state_exact(lib: OracleLib) -> None:
    """Row means of small integers: exact, equal on every row."""
    x = np.array([[1.0, 2.0, -3.0, 8.0], [3.0, -2.0, 5.0, 0.0], [5.0, 6.0, 1.0, -8.0], [-1.0, 2.0, 1.0, 4.0]])
    lib.average_state(x)
    assert np.array_equal(x, np.tile([[2.0, 2.0, 1.0, 1.0]], (4, 1)))


PINS = {
    "sgd_single_worker": pin_sgd_single_worker,
    "ddp_k1": pin_ddp_k1,
    "local_steps_independent": pin_local_steps_independent,
    "optimizer_state_stays_local": pin_optimizer_state_stays_local,
    "mean_gradient": pin_mean_gradient,
    "slowmo_geometric": pin_slowmo_geometric,
    "schedule_counts": pin_schedule_counts,
    "permutation_invariance": pin_permutation_invariance,
    "identical_replicas_identity": pin_identical_replicas_identity,
    "identical_gradients_match_local": pin_identical_gradients_match_local,
    "lr_schedule_vs_torch": pin_lr_schedule_vs_torch,
    "lr_schedule_closed_forms": pin_lr_schedule_closed_forms,
    "warmup_sync_counts": pin_warmup_sync_counts,
    "ddp_vs_torch": pin_ddp_vs_torch,
    "localsgd_vs_torch": pin_localsgd_vs_torch,
    "first_sync_linearity": pin_first_sync_linearity,
    "ddp_equals_cpdp_k1_beta0": pin_ddp_equals_cpdp_k1_beta0,
    "adamw_single_worker_vs_torch": pin_adamw_single_worker_vs_torch,
    "adamw_ddp_k1": pin_adamw_ddp_k1,
    "adamw_state_stays_local": pin_adamw_state_stays_local,
    "adamw_slowmo_geometric": pin_adamw_slowmo_geometric,
    "adamw_baselines_vs_torch": pin_adamw_baselines_vs_torch,
    "state_sync_vs_torch": pin_state_sync_vs_torch,
    "state_sync_makes_cpdp_k1_ddp": pin_state_sync_makes_cpdp_k1_ddp,
    "average_state_exact": pin_average_state_exact,
}
for _name in GOLDEN_CASES + METHOD_CASES:
    PINS[f"golden:{_name}"] = (lambda lib, _n=_name: pin_golden(lib, _n))


def failing_pins(lib: OracleLib) -> list[str]:
    """Names of the pins that this library fails."""
    failed = []
    for name, fn in PINS.items():
        try:
            fn(lib)
        except AssertionError:
            failed.append(name)
    return failed
