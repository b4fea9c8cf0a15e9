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
and v. The denominator is then max(|s_j|, rms_T(s), f_j), where the parameter
floor counts for at most 10 times the base denominator max(|s_j|, rms_T(s)):
the sensitivity of AdamW's direction has no upper bound, and the cap keeps
the check from accepting any value where it grows large.

The parameters also carry a history scale h_T: the largest rms_T of the
oracle's theta at any step so far, theta0 included. A float32 running update
theta -= lr * d rounds at every step relative to the value's magnitude then,
so the absolute error it carries is a few ulps of the largest magnitude the
value has had, not of its current one; where a tensor's values cancel toward
zero (a one-element tensor crossing zero, say), rms_T(s) shrinks and that
carried error becomes a large relative one. theta, theta_ref and v therefore
use max(|s_j|, rms_T(s), f_j, h_T) (h_T with no cap: it is a magnitude the
values have had, not a sensitivity).

run_and_check reports, beside the errors, the same metric with no floor at
all, the fraction of elements whose denominator a floor set, and the largest
floor-to-base ratio; the momentum-SGD checks of the named configurations and
the sweep points require the metric with no floor to meet the tolerance too.
"""
from __future__ import annotations

from dataclasses import dataclass

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


@dataclass
class ErrStats:
    """One state array's distance from the oracle.
    err: the metric with the floor (what the tolerance bounds);
    plain: the same metric with no floor at all;
    governed: elements whose denominator the floor set (floor above the base
    denominator max(|s_j|, rms_T(s))), out of count;
    max_ratio: the largest floor / base denominator over the array, before
    any cap."""
    err: float = 0.0
    plain: float = 0.0
    governed: int = 0
    count: int = 0
    max_ratio: float = 0.0


def error_stats(x, ref, tensor_id, scale=None, floor=None, cap=None, hist=None) -> ErrStats:
    """The error metric of the module docstring, per model tensor. With `cap`,
    the floor raises an element's denominator to at most cap times its base
    denominator. `hist` is the history scale of each column's tensor (no cap)."""
    x, ref = np.atleast_2d(x), np.atleast_2d(ref)
    s = ref if scale is None else np.broadcast_to(np.atleast_2d(scale), ref.shape)
    fl = None if floor is None else np.broadcast_to(np.atleast_2d(floor), ref.shape)
    hs = None if hist is None else np.broadcast_to(np.atleast_2d(hist), ref.shape)
    out = ErrStats(count=int(x.size))
    for t in np.unique(tensor_id):
        m = tensor_id == t
        sm = s[:, m]
        rms = float(np.sqrt(np.mean(sm * sm)))
        base = np.maximum(np.abs(sm), rms)
        if not np.any(base):
            base = np.ones_like(base)
        diff = np.abs(x[:, m] - ref[:, m])
        den = base
        raised = np.zeros(base.shape, dtype=bool)
        if fl is not None:
            f = fl[:, m]
            ratio = f / base
            raised |= ratio > 1.0
            out.max_ratio = max(out.max_ratio, float(np.max(ratio)))
            den = np.maximum(den, f if cap is None else np.minimum(f, cap * base))
        if hs is not None:
            h = hs[:, m]
            ratio = h / base
            raised |= ratio > 1.0
            out.max_ratio = max(out.max_ratio, float(np.max(ratio)))
            den = np.maximum(den, h)
        out.governed += int(np.count_nonzero(raised))
        out.err = max(out.err, float(np.max(diff / den)))
        out.plain = max(out.plain, float(np.max(diff / base)))
    return out


def scaled_error(x, ref, tensor_id, scale=None, floor=None) -> float:
    return error_stats(x, ref, tensor_id, scale, floor).err


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
                 device: str = "cuda", method: str = "cpdp", state_sync: bool = False, staging: int = 0,
                 shuffle: bool = False):
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
        self.gpu.set_reconcile_staging(staging)
        self.gpu.set_reconcile_shuffle(shuffle)
        self.orc = oracle.default()
        self.hp = oracle_hyper(wl)
        if self.adamw:
            self.algo = oracle.AdamWOracle(self.orc, f32(wl.adam_beta1), f32(wl.adam_beta2), f32(wl.adam_eps))
        else:
            self.algo = self.orc
        self.ost = self.algo.init(wl.W, self._host(theta0))
        self.floors = MomentFloors(self.orc, wl, self.adamw, method)
        self.tensors = np.unique(self.tensor_id)
        self.hist = np.zeros(len(self.tensors))  # each tensor's largest rms of theta so far
        self._grow_hist()
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
        self._grow_hist()
        return synced

    def _grow_hist(self) -> None:
        """The history scale: per tensor, the largest rms over all replicas that
        the oracle's theta has had at any step so far (theta0 included)."""
        for k, t in enumerate(self.tensors):
            th = self.ost.theta[:, self.tensor_id == t]
            self.hist[k] = max(self.hist[k], float(np.sqrt(np.mean(th * th))))

    # the parameter floor raises a denominator at most this many times over its base
    PARAM_FLOOR_CAP = 10.0

    def error_stats(self) -> dict[str, ErrStats]:
        """Every state array's ErrStats, plus "v_own_scale": v measured on its
        own scale (s = v) with no floor, for the record."""
        torch.cuda.synchronize(self.device)
        g = {k: self._host(getattr(self.gpu, k)) for k in ("params", "mom", "anchor", "slow_v")}
        o = self.ost
        tid = self.tensor_id
        pf, cap = self.floors.param, self.PARAM_FLOOR_CAP
        hist = self.hist[np.searchsorted(self.tensors, tid)]
        stats = {
            "theta": error_stats(g["params"], o.theta, tid, floor=pf, cap=cap, hist=hist),
            "buf": error_stats(g["mom"], o.buf, tid, floor=self.floors.floor["buf"]),
            "theta_ref": error_stats(g["anchor"], o.theta_ref, tid, floor=pf, cap=cap, hist=hist),
            "v": error_stats(g["slow_v"], o.v, tid, scale=o.theta_ref, floor=pf, cap=cap, hist=hist),
        }
        if self.adamw:
            stats["exp_avg_sq"] = error_stats(self._host(self.gpu.exp_avg_sq), o.sq, tid,
                                              floor=self.floors.floor["exp_avg_sq"])
        stats["v_own_scale"] = error_stats(g["slow_v"], o.v, tid)
        return stats

    def errors(self) -> dict[str, float]:
        return {k: v.err for k, v in self.error_stats().items() if k != "v_own_scale"}

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


class Worst(dict):
    """run_and_check's result: the worst error (with floors) per state array,
    and, over all steps and arrays, the worst error with no floor (`plain`),
    v's worst error on its own scale (`v_own_scale`), the largest fraction of
    an array's elements whose denominator a floor set (`governed_frac`) and
    the largest floor / base denominator ratio (`max_floor_ratio`)."""
    plain = 0.0
    v_own_scale = 0.0
    governed_frac = 0.0
    max_floor_ratio = 0.0


def run_and_check(wl: wls.Workload, cols=None, tol: float = TOL, seed: int = 42,
                  steps: int | None = None, method: str = "cpdp", state_sync: bool = False,
                  staging: int = 0, shuffle: bool = False, plain: bool = False) -> Worst:
    """Run an epoch (or `steps` steps) of `method` on both sides, checking every
    step. With `plain`, the metric with no floor must meet `tol` too."""
    pair = Pair(wl, cols, seed, method=method, state_sync=state_sync, staging=staging, shuffle=shuffle)
    worst = Worst()
    try:
        for t in range(1, (steps or wl.T) + 1):
            synced = pair.step(t)
            stats = pair.error_stats()
            worst.v_own_scale = max(worst.v_own_scale, stats.pop("v_own_scale").plain)
            for k, st in stats.items():
                worst[k] = max(worst.get(k, 0.0), st.err)
                worst.plain = max(worst.plain, st.plain)
                worst.governed_frac = max(worst.governed_frac, st.governed / max(1, st.count))
                worst.max_floor_ratio = max(worst.max_floor_ratio, st.max_ratio)
                assert st.err <= tol, f"{wl.name} t={t}: {k} error {st.err:.3e} > {tol:.0e} ({stats})"
                if plain:
                    assert st.plain <= tol, f"{wl.name} t={t}: {k} error without floor {st.plain:.3e} > {tol:.0e}"
            if synced:
                assert pair.replicas_identical(), f"{wl.name} t={t}: replicas differ after reconcile"
    finally:
        pair.close()
    return worst
