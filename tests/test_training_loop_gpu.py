"""CPDP driving a real (small) model: W workers each hold an MLP whose
parameters are views into their row of the [W][N] replica buffer, compute
gradients with autograd on their own data shard into the [W][N] gradient
buffer, and step through the library with the paper's protocol (a warmup
epoch at K = 1, then K = 2, cosine learning rate, SlowMo beta = 0.3), with
momentum SGD, with AdamW (the paper's ViT-S optimizer), and with AdamW plus
optimizer-state reconciliation. Every step is checked
against the fp64 oracle fed the same gradients (the gradients are inputs of
the method), the replicas must be bit-identical after every synchronization,
and the training loss must fall."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2607_21224_gb300 import workloads as wls
from paper_2607_21224_gb300.state import CPDPState
from parity import TOL, MomentFloors, scaled_error

pytestmark = pytest.mark.gpu

SHAPES = [(64, 16), (64,), (32, 64), (32,), (1, 32), (1,)]


def views(row: torch.Tensor):
    """Parameter tensors laid out back to back in one flat row."""
    out, o = [], 0
    for s in SHAPES:
        n = math.prod(s)
        out.append(row[o:o + n].view(s))
        o += n
    return out


def mlp(params, x):
    w1, b1, w2, b2, w3, b3 = params
    h = torch.tanh(x @ w1.T + b1)
    h = torch.tanh(h @ w2.T + b2)
    return (h @ w3.T + b3).squeeze(-1)


@pytest.mark.parametrize("opt,state_sync", [("sgd", False), ("adamw", False), ("adamw", True)])
def test_cpdp_trains_an_mlp_with_oracle_parity(opt, state_sync):
    dev = torch.device("cuda")
    W, K, T, E, We = 4, 2, 16, 4, 1
    N = sum(math.prod(s) for s in SHAPES)
    gen = torch.Generator(device="cpu").manual_seed(0)
    # data: a fixed teacher network, each worker with its own shard and batches
    teacher = torch.randn(N, generator=gen) * 0.2
    X = torch.randn(W, E * T, 32, 16, generator=gen)
    Y = torch.stack([mlp(views(teacher), X[i].reshape(-1, 16)).reshape(E * T, 32) for i in range(W)])
    X, Y = X.to(dev), Y.to(dev)
    theta0 = (torch.randn(N, generator=gen) * 0.1).to(dev)

    beta = 0.3  # the paper's SlowMo setting (Table 3)
    if opt == "adamw":  # decoupled decay; lr and minimum chosen so the loss falls ~10x in four epochs
        lr, min_lr, mu, wd = 3e-3, 6e-5, 0.0, 1e-2
    else:
        lr, min_lr, mu, wd = 0.02, 1e-3, 0.9, 1e-4
    f = lambda x: float(np.float32(x))  # noqa: E731
    hp = oracle.Hyper(lr=f(lr), momentum=f(mu), weight_decay=f(wd), K=K, beta=f(beta), alpha=1.0)
    orc = oracle.default()
    algo = oracle.AdamWOracle(orc, f(0.9), f(0.999), f(1e-8)) if opt == "adamw" else orc
    wl = wls.Workload("mlp", W=W, tensors=tuple(wls.flat_tensors(N)), K=K, T=T, momentum=mu, beta=beta,
                      optimizer=opt)
    floors = MomentFloors(orc, wl, opt == "adamw", "cpdp")
    grads = torch.empty((W, N), device=dev)
    tid = np.searchsorted(np.cumsum([0] + [math.prod(s) for s in SHAPES]), np.arange(N), side="right") - 1
    losses = []
    with CPDPState(W, N, lr=lr, momentum=mu, weight_decay=wd, K=K, beta=beta) as st:
        if opt == "adamw":
            st.set_adamw()
        st.set_state_reconcile(state_sync)
        st.init_params(theta0)
        st.set_schedule(T, E, We, lr, min_lr)
        ost = algo.init(W, theta0.double().cpu().numpy())
        for e in range(E):
            epoch_loss = 0.0
            for t in range(1, T + 1):
                b = e * T + t - 1
                for i in range(W):
                    p = [v.detach().requires_grad_(True) for v in views(st.params[i])]
                    loss = torch.mean((mlp(p, X[i, b]) - Y[i, b]) ** 2)
                    gs = torch.autograd.grad(loss, p)
                    grads[i].copy_(torch.cat([g.reshape(-1) for g in gs]))
                    epoch_loss += loss.item() / (W * T)
                synced = st.step_at(grads, e, t)
                hp.lr = f(orc.scheduled_lr(f(lr), f(min_lr), We * T, E * T, b))
                g_host = grads.double().cpu().numpy()
                want = orc.is_sync_step_at(e, t, K, T, We)
                assert synced == want
                (algo.reconcile if want else algo.local_step)(ost, g_host, hp)
                floors.update(ost, g_host, want, True, state_sync, hp.lr)
                torch.cuda.synchronize()
                checks = [("theta", st.params, ost.theta, floors.param), ("theta_ref", st.anchor, ost.theta_ref, floors.param),
                          ("buf", st.mom, ost.buf, floors.floor["buf"])]
                if opt == "adamw":
                    checks.append(("exp_avg_sq", st.exp_avg_sq, ost.sq, floors.floor["exp_avg_sq"]))
                for key, x, ref, floor in checks:
                    err = scaled_error(x.double().cpu().numpy(), ref, tid, floor=floor)
                    assert err <= TOL, (e, t, key, err)
                assert scaled_error(st.slow_v.double().cpu().numpy(), ost.v, tid, scale=ost.theta_ref,
                                    floor=floors.param) <= TOL
                if synced:
                    p = st.params.view(torch.int32)
                    assert torch.equal(p, p[0:1].expand_as(p))
            losses.append(epoch_loss)
    assert losses[-1] < 0.25 * losses[0], losses
