"""fp64 CPU oracle for CPDP's data-parallel hot path.

TEST INFRASTRUCTURE. Only the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference arm import this package. The product path
(the CUDA library and its binding) never imports it and shares no code with it.

The arithmetic lives in ``cpdp_oracle.c`` (plain C, double precision,
single-threaded); this module compiles it with gcc and marshals numpy float64
arrays to it. It follows Algorithm 1 of the paper (CPDP with SlowMo momentum)
with the momentum-SGD optimizer step of Sec. 4.2 / Table 3; see the header of
``cpdp_oracle.c`` for the formulas and their citations.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
SOURCE = _HERE / "cpdp_oracle.c"
LIBRARY = _HERE / "libcpdp_oracle.so"
# No fused multiply-add and no fast-math: each operation rounds once, in fp64.
CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]


def build_oracle(source: Path = SOURCE, output: Path = LIBRARY, force: bool = False) -> Path:
    """Compile the oracle C source into a shared library with gcc."""
    source, output = Path(source), Path(output)
    if not force and output.exists() and output.stat().st_mtime >= source.stat().st_mtime:
        return output
    tmp = output.with_suffix(f".{os.getpid()}.tmp")
    subprocess.run(["gcc", *CFLAGS, "-o", str(tmp), str(source), "-lm"], check=True)
    os.replace(tmp, output)
    return output


_f64p = ctypes.POINTER(ctypes.c_double)


def _ptr(a: np.ndarray):
    assert a.dtype == np.float64 and a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(_f64p)


class OracleLib:
    """ctypes view of one compiled oracle library (the real one, or a test mutant)."""

    def __init__(self, path: Path | str | None = None):
        if path is None:
            path = build_oracle()
        self.path = Path(path)
        lib = ctypes.CDLL(str(self.path))
        i64, c_int, dbl = ctypes.c_int64, ctypes.c_int, ctypes.c_double
        lib.oracle_init.argtypes = [c_int, i64, _f64p, _f64p, _f64p, _f64p, _f64p]
        lib.oracle_init.restype = None
        lib.oracle_local_step.argtypes = [c_int, i64, dbl, dbl, dbl, _f64p, _f64p, _f64p]
        lib.oracle_local_step.restype = None
        lib.oracle_reconcile.argtypes = [c_int, i64, dbl, dbl, dbl, dbl, dbl,
                                         _f64p, _f64p, _f64p, _f64p, _f64p]
        lib.oracle_reconcile.restype = c_int
        lib.oracle_is_sync_step.argtypes = [i64, i64, i64]
        lib.oracle_is_sync_step.restype = c_int
        lib.oracle_scheduled_lr.argtypes = [dbl, dbl, i64, i64, i64]
        lib.oracle_scheduled_lr.restype = dbl
        lib.oracle_is_sync_step_at.argtypes = [i64, i64, i64, i64, i64]
        lib.oracle_is_sync_step_at.restype = c_int
        lib.oracle_localsgd_sync.argtypes = [c_int, i64, dbl, dbl, dbl, _f64p, _f64p, _f64p]
        lib.oracle_localsgd_sync.restype = c_int
        lib.oracle_ddp_step.argtypes = [c_int, i64, dbl, dbl, dbl, _f64p, _f64p, _f64p]
        lib.oracle_ddp_step.restype = c_int
        lib.oracle_adamw_local_step.argtypes = [c_int, i64, dbl, dbl, dbl, dbl, dbl, i64,
                                                _f64p, _f64p, _f64p, _f64p]
        lib.oracle_adamw_local_step.restype = None
        lib.oracle_adamw_reconcile.argtypes = [c_int, i64, dbl, dbl, dbl, dbl, dbl, i64, dbl, dbl,
                                               _f64p, _f64p, _f64p, _f64p, _f64p, _f64p]
        lib.oracle_adamw_reconcile.restype = c_int
        lib.oracle_average_state.argtypes = [c_int, i64, _f64p]
        lib.oracle_average_state.restype = c_int
        for name in ("oracle_adamw_localsgd_sync", "oracle_adamw_ddp_step"):
            getattr(lib, name).argtypes = [c_int, i64, dbl, dbl, dbl, dbl, dbl, i64, _f64p, _f64p, _f64p, _f64p]
            getattr(lib, name).restype = c_int
        self._lib = lib

    # -- Algorithm 1 pieces -------------------------------------------------
    def init(self, W: int, theta0: np.ndarray) -> "OracleState":
        theta0 = np.ascontiguousarray(theta0, dtype=np.float64).reshape(-1)
        N = theta0.size
        st = OracleState(theta=np.empty((W, N)), buf=np.empty((W, N)),
                         theta_ref=np.empty(N), v=np.empty(N))
        self._lib.oracle_init(W, N, _ptr(theta0), _ptr(st.theta), _ptr(st.buf),
                              _ptr(st.theta_ref), _ptr(st.v))
        return st

    def local_step(self, st: "OracleState", g: np.ndarray, hp: "Hyper") -> None:
        g = _grads(g, st)
        W, N = st.theta.shape
        self._lib.oracle_local_step(W, N, hp.lr, hp.momentum, hp.weight_decay,
                                    _ptr(g), _ptr(st.theta), _ptr(st.buf))

    def reconcile(self, st: "OracleState", g: np.ndarray, hp: "Hyper") -> None:
        g = _grads(g, st)
        W, N = st.theta.shape
        rc = self._lib.oracle_reconcile(W, N, hp.lr, hp.momentum, hp.weight_decay,
                                        hp.beta, hp.alpha, _ptr(g), _ptr(st.theta),
                                        _ptr(st.buf), _ptr(st.theta_ref), _ptr(st.v))
        if rc != 0:
            raise MemoryError("oracle_reconcile could not allocate its temporaries")

    def is_sync_step(self, t: int, K: int, T: int) -> bool:
        return bool(self._lib.oracle_is_sync_step(t, K, T))

    def scheduled_lr(self, base_lr: float, min_lr: float, warmup_steps: int, total_steps: int,
                     s: int) -> float:
        return float(self._lib.oracle_scheduled_lr(base_lr, min_lr, warmup_steps, total_steps, s))

    def is_sync_step_at(self, epoch: int, t: int, K: int, T: int, warmup_epochs: int) -> bool:
        return bool(self._lib.oracle_is_sync_step_at(epoch, t, K, T, warmup_epochs))

    def localsgd_sync(self, st: "OracleState", g: np.ndarray, hp: "Hyper") -> None:
        g = _grads(g, st)
        W, N = st.theta.shape
        if self._lib.oracle_localsgd_sync(W, N, hp.lr, hp.momentum, hp.weight_decay, _ptr(g),
                                          _ptr(st.theta), _ptr(st.buf)) != 0:
            raise MemoryError("oracle_localsgd_sync could not allocate")

    def ddp_step(self, st: "OracleState", g: np.ndarray, hp: "Hyper") -> None:
        g = _grads(g, st)
        W, N = st.theta.shape
        if self._lib.oracle_ddp_step(W, N, hp.lr, hp.momentum, hp.weight_decay, _ptr(g),
                                     _ptr(st.theta), _ptr(st.buf)) != 0:
            raise MemoryError("oracle_ddp_step could not allocate")

    def average_state(self, state: np.ndarray) -> None:
        """Replace every worker's row of a [W][N] state array by the row mean."""
        W, N = state.shape
        if self._lib.oracle_average_state(W, N, _ptr(state)) != 0:
            raise MemoryError("oracle_average_state could not allocate")

    def step(self, st: "OracleState", g: np.ndarray, hp: "Hyper", t: int, T: int,
             method: str = "cpdp", state_sync: bool = False) -> bool:
        """One mini-batch step t (1-based) of an epoch of T steps of `method`
        ("cpdp", "localsgd" or "ddp"); returns whether it synchronized. With
        state_sync, a CPDP or LocalSGD synchronization also averages the
        momentum buffers over the workers."""
        if method == "ddp":
            self.ddp_step(st, g, hp)
            return True
        if self.is_sync_step(t, hp.K, T):
            (self.localsgd_sync if method == "localsgd" else self.reconcile)(st, g, hp)
            if state_sync:
                self.average_state(st.buf)
            return True
        self.local_step(st, g, hp)
        return False


class AdamWOracle:
    """The same Algorithm 1 with AdamW as each worker's optimizer. State: the
    OracleState's buf is the first moment m; `sq` holds the second moments.
    The optimizer step counter is shared by all workers (every worker steps at
    every mini-batch) and advanced by each local step or reconcile."""

    def __init__(self, lib: OracleLib, beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8):
        self.lib, self.beta1, self.beta2, self.eps = lib, beta1, beta2, eps

    def init(self, W: int, theta0: np.ndarray) -> "OracleState":
        st = self.lib.init(W, theta0)
        st.sq = np.zeros_like(st.buf)
        st.opt_step = 0
        return st

    def local_step(self, st: "OracleState", g: np.ndarray, hp: "Hyper") -> None:
        g = _grads(g, st)
        W, N = st.theta.shape
        st.opt_step += 1
        self.lib._lib.oracle_adamw_local_step(W, N, hp.lr, self.beta1, self.beta2, self.eps, hp.weight_decay,
                                              st.opt_step, _ptr(g), _ptr(st.theta), _ptr(st.buf), _ptr(st.sq))

    def reconcile(self, st: "OracleState", g: np.ndarray, hp: "Hyper") -> None:
        g = _grads(g, st)
        W, N = st.theta.shape
        st.opt_step += 1
        rc = self.lib._lib.oracle_adamw_reconcile(W, N, hp.lr, self.beta1, self.beta2, self.eps,
                                                  hp.weight_decay, st.opt_step, hp.beta, hp.alpha, _ptr(g),
                                                  _ptr(st.theta), _ptr(st.buf), _ptr(st.sq),
                                                  _ptr(st.theta_ref), _ptr(st.v))
        if rc != 0:
            raise MemoryError("oracle_adamw_reconcile could not allocate")

    def _baseline(self, name: str, st: "OracleState", g: np.ndarray, hp: "Hyper") -> None:
        g = _grads(g, st)
        W, N = st.theta.shape
        st.opt_step += 1
        if getattr(self.lib._lib, name)(W, N, hp.lr, self.beta1, self.beta2, self.eps, hp.weight_decay,
                                        st.opt_step, _ptr(g), _ptr(st.theta), _ptr(st.buf), _ptr(st.sq)) != 0:
            raise MemoryError(f"{name} could not allocate")

    def step(self, st: "OracleState", g: np.ndarray, hp: "Hyper", t: int, T: int,
             method: str = "cpdp", state_sync: bool = False) -> bool:
        if method == "ddp":
            self._baseline("oracle_adamw_ddp_step", st, g, hp)
            return True
        if self.lib.is_sync_step(t, hp.K, T):
            if method == "localsgd":
                self._baseline("oracle_adamw_localsgd_sync", st, g, hp)
            else:
                self.reconcile(st, g, hp)
            if state_sync:
                self.lib.average_state(st.buf)
                self.lib.average_state(st.sq)
            return True
        self.local_step(st, g, hp)
        return False


def _grads(g: np.ndarray, st: "OracleState") -> np.ndarray:
    g = np.ascontiguousarray(g, dtype=np.float64)
    if g.shape != st.theta.shape:
        raise ValueError(f"grads shape {g.shape} != state shape {st.theta.shape}")
    return g


@dataclass
class Hyper:
    """Hyperparameters of one run: lr (eta), momentum (mu), weight_decay
    (lambda), sync period K, SlowMo beta, and outer step alpha (1 = paper)."""
    lr: float
    momentum: float
    weight_decay: float
    K: int
    beta: float
    alpha: float = 1.0


@dataclass
class OracleState:
    """theta and buf are (W, N); theta_ref and v are (N,). All float64."""
    theta: np.ndarray
    buf: np.ndarray
    theta_ref: np.ndarray
    v: np.ndarray

    def copy(self) -> "OracleState":
        return OracleState(self.theta.copy(), self.buf.copy(), self.theta_ref.copy(), self.v.copy())


_default: OracleLib | None = None


def default() -> OracleLib:
    """The oracle built from this package's source (compiled on first use)."""
    global _default
    if _default is None:
        _default = OracleLib()
    return _default
