"""Drive the CUDA path (through the C ABI) and the fp64 oracle on the same
seeded inputs, and measure how far apart they are.

Every parameter column j of CPDP is an independent problem (the update is
elementwise in j; the only reduction is over the W workers of one column), so
the oracle can run on any subset of columns and its result is exactly what it
would compute for those columns inside the full problem. Full-size workloads
are therefore checked on windows of columns: the head, every tensor boundary
the window set includes, the ragged tail, and random columns.

Error metric (the tolerance reading for "max relative error 1e-5"): for each
model tensor T and state array x with oracle value r and scale s,
    err = max_j |x_j - r_j| / max(|s_j|, rms_T(s)),
with s = r for theta (all replicas), theta_ref and buf, and s = theta_ref for
the SlowMo velocity v. v = beta v + (theta_avg - theta_ref) is a difference of
two parameter-sized float32 numbers, so its rounding error is a few float32
ulps of the parameters, not of v; it is measured in parameter units.

Means over the W workers get the same treatment. A float32 sum of W terms is
accurate to a few ulps of the mean of the terms' magnitudes, not of the mean
itself, which cancellation can make far smaller. So each moment array (buf;
AdamW's second moments) also carries a floor f_j under its scale: at a step
that forms a mean over the workers, f_j grows by the magnitude of what was
averaged (the gradients' mean |g_ij| times the mean gradient's coefficient in
the moment; at a state-reconciling sync, the mean |state_ij| of the states
averaged), and every step carries it forward with the moment's own decay
factor (momentum, beta1 or beta2), as the recurrence carries the error.
The parameters carry a floor too. Each step moves them by lr times the
optimizer's direction (buf for SGD, m^/(sqrt(v^) + eps) for AdamW), whose
error is at most the direction's sensitivity to the moments times their
floors. AdamW's direction is ill-conditioned where a mean gradient cancels to
near eps: at its first step it is lr * g/(|g| + eps). The parameter floor sums
lr times those sensitivities times the moment floors, scaled by what SlowMo can
carry into theta_ref and v (1 + alpha/(1 - beta)). It serves theta, theta_ref
and v. The denominator is then max(|s_j|, rms_T(s), f_j).
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2607_21224_gb300 import workloads as wls
from paper_2607_21224_gb300.state import CPDPState

TOL = 1e-5


def f32(x: float) -> float:
    """The float32 value the C ABI receives for a Python float."""
    return float(np.float32(x))


def oracle_hyper(wl: wls.Workload) -> oracle.Hyper:
    return oracle.Hyper(lr=f32(wl.lr), momentum=f32(wl.momentum), weight_decay=f32(wl.weight_decay),
                        K=wl.K, beta=f32(wl.beta), alpha=f32(wl.alpha))


def scaled_error(x, ref, tensor_id, scale=None, floor=None) -> float:
    x, ref = np.atleast_2d(x), np.atleast_2d(ref)
    s = ref if scale is None else np.broadcast_to(np.atleast_2d(scale), ref.shape)
    fl = None if floor is None else np.broadcast_to(np.atleast_2d(floor), ref.shape)
    worst = 0.0
    for t in np.unique(tensor_id):
        m = tensor_id == t
        sm = s[:, m]
        rms = float(np.sqrt(np.mean(sm * sm)))
        den = np.maximum(np.abs(sm), rms)
        if fl is not None:
            den = np.maximum(den, fl[:, m])
        if not np.any(den):
            den = np.ones_like(den)
        worst = max(worst, float(np.max(np.abs(x[:, m] - ref[:, m]) / den)))
    return worst


def windows(wl: wls.Workload, width: int = 2048, n_random: int = 2048, seed: int = 0,
            boundaries: int = 12) -> np.ndarray:
    """Column indices: head, tail, `boundaries` tensor boundaries spread over
    the model (width//8 columns each side), and random columns."""
    N, offs = wl.N, wl.offsets
    cols = [np.arange(0, min(width, N)), np.arange(max(0, N - width - 3), N)]
    inner = offs[1:-1]
    if inner:
        pick = np.unique(np.linspace(0, len(inner) - 1, min(boundaries, len(inner))).astype(int))
        for k in pick:
            b = inner[k]
            cols.append(np.arange(max(0, b - width // 8), min(N, b + width // 8)))
    rng = np.random.default_rng(seed)
    cols.append(rng.integers(0, N, n_random))
    return np.unique(np.concatenate(cols)).astype(np.int64)


class MomentFloors:
    """Error floors (module docstring) of the moment arrays (buf; AdamW's
    second moments) and of the parameters (theta, theta_ref, v). update()
    follows one oracle step that was run without its state average. It grows
    the moment floors by what this step averaged over the workers and decays
    them by each moment's own factor. It grows the parameter floor by lr times
    the step direction's sensitivity to the moment floors, times what SlowMo
    can carry into theta_ref and v. Last, it applies the oracle's state average
    when the step reconciles states."""

    def __init__(self, orc, wl: wls.Workload, adamw: bool, method: str = "cpdp"):
        self.orc, self.adamw = orc, adamw
        self.beta1, self.beta2, self.eps = f32(wl.adam_beta1), f32(wl.adam_beta2), f32(wl.adam_eps)
        self.carry = ({"buf": self.beta1, "exp_avg_sq": self.beta2} if adamw else {"buf": f32(wl.momentum)})
        self.floor = {k: 0.0 for k in self.carry}
        self.param = 0.0
        # an error in theta reaches theta_ref and v through SlowMo at most alpha / (1 - beta) times over
        self.slowmo = 1.0 + (f32(wl.alpha) / (1.0 - f32(wl.beta)) if method == "cpdp" else 0.0)

    def update(self, ost, g: np.ndarray, synced: bool, used_gbar: bool, state_sync: bool, lr: float) -> None:
        added = {k: 0.0 for k in self.carry}
        if synced and used_gbar:  # this step used the gradient mean
            gmag = np.abs(g).mean(axis=0)
            if self.adamw:
                added["buf"] = (1.0 - self.beta1) * gmag
                added["exp_avg_sq"] = (1.0 - self.beta2) * 2.0 * np.abs(g.mean(axis=0)) * gmag
            else:
                added["buf"] = gmag
        if synced and state_sync:
            added["buf"] = added["buf"] + np.abs(ost.buf).mean(axis=0)
            if self.adamw:
                added["exp_avg_sq"] = added["exp_avg_sq"] + np.abs(ost.sq).mean(axis=0)
        for k, c in self.carry.items():
            self.floor[k] = added[k] + c * self.floor[k]
        # this step's parameter update: lr * buf (SGD) or lr * m^/(sqrt(v^) + eps) (AdamW),
        # with the per-worker states the step used (before any state average)
        if self.adamw:
            t = ost.opt_step
            bc1, bc2 = 1.0 - self.beta1 ** t, 1.0 - self.beta2 ** t
            root = np.sqrt(ost.sq / bc2)
            den = root + self.eps
            sens_m = 1.0 / (bc1 * den)
            sens_v = (np.abs(ost.buf) / bc1) / (2.0 * bc2 * np.maximum(root, self.eps) * den * den)
            inc = lr * (sens_m.max(axis=0) * self.floor["buf"] + sens_v.max(axis=0) * self.floor["exp_avg_sq"])
        else:
            inc = lr * self.floor["buf"]
        self.param = self.param + self.slowmo * inc
        if synced and state_sync:
            self.orc.average_state(ost.buf)
            if self.adamw:
                self.orc.average_state(ost.sq)


class Pair:
    """A CPDPState on the GPU and an oracle state over `cols` (all if None)."""

    def __init__(self, wl: wls.Workload, cols: np.ndarray | None = None, seed: int = 42,
                 device: str = "cuda", method: str = "cpdp", state_sync: bool = False):
        self.wl, self.seed, self.device, self.method = wl, seed, torch.device(device), method
        self.state_sync = state_sync
        self.cols = np.arange(wl.N, dtype=np.int64) if cols is None else np.asarray(cols, np.int64)
        self.full = cols is None
        self.cols_dev = torch.from_numpy(self.cols).to(self.device)
        self.tensor_id = np.searchsorted(np.asarray(wl.offsets), self.cols, side="right") - 1
        theta0 = wls.make_theta0(wl, seed, self.device)
        self.gpu = CPDPState(wl.W, wl.N, wl.offsets, device=self.device, **wl.hyper())
        self.adamw = wl.optimizer == "adamw"
        if self.adamw:
            self.gpu.set_adamw(wl.adam_beta1, wl.adam_beta2, wl.adam_eps)
        self.gpu.init_params(theta0)
        self.gpu.set_method(method)
        self.gpu.set_state_reconcile(state_sync)
        self.orc = oracle.default()
        self.hp = oracle_hyper(wl)
        if self.adamw:
            self.algo = oracle.AdamWOracle(self.orc, f32(wl.adam_beta1), f32(wl.adam_beta2), f32(wl.adam_eps))
        else:
            self.algo = self.orc
        self.ost = self.algo.init(wl.W, self._host(theta0))
        self.floors = MomentFloors(self.orc, wl, self.adamw, method)
        self.grads = torch.empty((wl.W, wl.N), dtype=wl.torch_grad_dtype, device=self.device)

    def _host(self, t: torch.Tensor) -> np.ndarray:
        sel = t if self.full else t.index_select(t.dim() - 1, self.cols_dev)
        return sel.float().double().cpu().numpy()

    def step(self, t: int) -> bool:
        wls.make_grads(self.wl, t, self.seed, self.device, out=self.grads)
        synced = self.gpu.step(self.grads, t, self.wl.T)
        g = self._host(self.grads)
        # the oracle's step without its state average, which the floors apply
        o_synced = self.algo.step(self.ost, g, self.hp, t, self.wl.T, self.method, False)
        assert synced == o_synced, f"t={t}: GPU sync={synced}, oracle sync={o_synced}"
        self.floors.update(self.ost, g, o_synced, self.method != "localsgd", self.state_sync, self.hp.lr)
        return synced

    def errors(self) -> dict[str, float]:
        torch.cuda.synchronize(self.device)
        g = {k: self._host(getattr(self.gpu, k)) for k in ("params", "mom", "anchor", "slow_v")}
        o = self.ost
        tid = self.tensor_id
        errs = {
            "theta": scaled_error(g["params"], o.theta, tid, floor=self.floors.param),
            "buf": scaled_error(g["mom"], o.buf, tid, floor=self.floors.floor["buf"]),
            "theta_ref": scaled_error(g["anchor"], o.theta_ref, tid, floor=self.floors.param),
            "v": scaled_error(g["slow_v"], o.v, tid, scale=o.theta_ref, floor=self.floors.param),
        }
        if self.adamw:
            errs["exp_avg_sq"] = scaled_error(self._host(self.gpu.exp_avg_sq), o.sq, tid,
                                              floor=self.floors.floor["exp_avg_sq"])
        return errs

    def replicas_identical(self) -> bool:
        """After a synchronization: all W full rows bit-identical, and (CPDP) the
        anchor equal to row 0 bit for bit (checked on the whole arrays, any size)."""
        p = self.gpu.params.view(torch.int32)
        same = bool(torch.equal(p, p[0:1].expand_as(p)))
        if self.method == "cpdp":
            same = same and bool(torch.equal(p[0], self.gpu.anchor.view(torch.int32)))
        if self.state_sync or self.method == "ddp":
            states = [self.gpu.mom] + ([self.gpu.exp_avg_sq] if self.adamw else [])
            for x in states:
                b = x.view(torch.int32)
                same = same and bool(torch.equal(b, b[0:1].expand_as(b)))
        return same

    def close(self):
        self.gpu.close()


def run_and_check(wl: wls.Workload, cols=None, tol: float = TOL, seed: int = 42,
                  steps: int | None = None, method: str = "cpdp", state_sync: bool = False) -> dict[str, float]:
    """Run an epoch (or `steps` steps) of `method` on both sides, checking every step."""
    pair = Pair(wl, cols, seed, method=method, state_sync=state_sync)
    worst: dict[str, float] = {}
    try:
        for t in range(1, (steps or wl.T) + 1):
            synced = pair.step(t)
            errs = pair.errors()
            for k, e in errs.items():
                worst[k] = max(worst.get(k, 0.0), e)
                assert e <= tol, f"{wl.name} t={t}: {k} error {e:.3e} > {tol:.0e} ({errs})"
            if synced:
                assert pair.replicas_identical(), f"{wl.name} t={t}: replicas differ after reconcile"
    finally:
        pair.close()
    return worst
