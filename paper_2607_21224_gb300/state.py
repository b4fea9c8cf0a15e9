"""CPDP state on one GPU: torch tensors for device memory and streams, libcpdp
for every step of the path.

``CPDPState`` owns the four state buffers of the C ABI's layout (replicas and
momentum buffers [W][N], anchor and SlowMo velocity [N], all float32) and calls
the binding in ``cpdp.py``. Torch only allocates memory and supplies streams.
"""
from __future__ import annotations

import torch

from . import cpdp as _c


def grad_dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return _c.CPDP_F32
    if t.dtype == torch.bfloat16:
        return _c.CPDP_BF16
    raise TypeError(f"gradients must be float32 or bfloat16, got {t.dtype}")


class CPDPState:
    """W simulated workers' replicas of an N-parameter model (Algorithm 1)."""

    def __init__(self, W: int, N: int, tensor_offsets=None, *, lr: float, momentum: float,
                 weight_decay: float, K: int, beta: float, alpha: float = 1.0, device="cuda"):
        self.W, self.N = int(W), int(N)
        self.device = torch.device(device)
        if self.device.type != "cuda":
            raise ValueError("CPDPState lives on a CUDA device; there is no CPU implementation")
        self.ctx = _c.cpdp_create(W, N, tensor_offsets, lr, momentum, weight_decay, K, beta, alpha)
        try:
            kw = dict(dtype=torch.float32, device=self.device)
            self.params = torch.empty((self.W, self.N), **kw)
            self.mom = torch.empty((self.W, self.N), **kw)
            self.anchor = torch.empty(self.N, **kw)
            self.slow_v = torch.empty(self.N, **kw)
            _c.cpdp_bind(self.ctx, self.params, self.mom, self.anchor, self.slow_v)
        except BaseException:
            _c.cpdp_destroy(self.ctx)
            self.ctx = None
            raise
        self.K = int(K)

    # -- plumbing ----------------------------------------------------------
    def _stream(self, stream) -> int:
        if stream is None:
            stream = torch.cuda.current_stream(self.device)
        return stream if isinstance(stream, int) else stream.cuda_stream

    def _grads(self, grads: torch.Tensor) -> torch.Tensor:
        if tuple(grads.shape) != (self.W, self.N) or not grads.is_contiguous():
            raise ValueError(f"grads must be a contiguous ({self.W}, {self.N}) tensor, got "
                             f"{tuple(grads.shape)} contiguous={grads.is_contiguous()}")
        if grads.device.type == "cpu" and not grads.is_pinned():
            raise ValueError("host gradients must be in page-locked (pinned) memory")
        return grads

    # -- the path ----------------------------------------------------------
    def init_params(self, theta0: torch.Tensor, stream=None) -> None:
        if theta0.dtype != torch.float32 or theta0.numel() != self.N or not theta0.is_contiguous():
            raise ValueError("theta0 must be a contiguous float32 tensor of N elements")
        if theta0.device.type == "cpu" and not theta0.is_pinned():
            raise ValueError("a host theta0 must be in page-locked (pinned) memory")
        _c.cpdp_init_params(self.ctx, theta0, self._stream(stream))

    def local_step(self, grads: torch.Tensor, stream=None) -> None:
        g = self._grads(grads)
        _c.cpdp_local_step(self.ctx, g, grad_dtype_code(g), self._stream(stream))

    def reconcile(self, grads: torch.Tensor, stream=None) -> None:
        g = self._grads(grads)
        _c.cpdp_reconcile(self.ctx, g, grad_dtype_code(g), self._stream(stream))

    def is_sync_step(self, t: int, steps_per_epoch: int) -> bool:
        r = _c.cpdp_is_sync_step(self.ctx, t, steps_per_epoch)
        if r < 0:
            raise ValueError(f"invalid step t={t} for an epoch of {steps_per_epoch} steps")
        return bool(r)

    def step(self, grads: torch.Tensor, t: int, steps_per_epoch: int, stream=None) -> bool:
        g = self._grads(grads)
        return _c.cpdp_step(self.ctx, g, grad_dtype_code(g), t, steps_per_epoch, self._stream(stream))

    def set_lr(self, lr: float) -> None:
        _c.cpdp_set_lr(self.ctx, lr)

    def set_adamw(self, beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8) -> None:
        """Switch the workers' optimizer to AdamW: lr and weight_decay given at
        creation become AdamW's lr and decoupled weight decay; `mom` holds the
        first moments and a new [W][N] tensor `exp_avg_sq` the second. Call it
        before init_params, which zeroes both moments and the step count."""
        if getattr(self, "exp_avg_sq", None) is None:
            self.exp_avg_sq = torch.zeros((self.W, self.N), dtype=torch.float32, device=self.device)
        _c.cpdp_set_adamw(self.ctx, beta1, beta2, eps, self.exp_avg_sq)

    @property
    def optimizer_step(self) -> int:
        return _c.cpdp_get_optimizer_step(self.ctx)

    @optimizer_step.setter
    def optimizer_step(self, step: int) -> None:
        _c.cpdp_set_optimizer_step(self.ctx, step)

    def set_state_reconcile(self, enable: bool) -> None:
        """Average the workers' optimizer states at every CPDP/LocalSGD sync
        (the variant the paper names but does not use); default off."""
        _c.cpdp_set_state_reconcile(self.ctx, enable)

    def set_pdl(self, enable: bool) -> None:
        """Programmatic dependent launch of the kernels (default on; results
        are bit-identical either way)."""
        _c.cpdp_set_pdl(self.ctx, enable)

    def set_reconcile_staging(self, stages: int) -> None:
        """0 (default): the reconcile loads its rows directly; 2..8: rows
        staged through that many shared-memory slots by bulk copies (the
        measured alternative; bit-identical results)."""
        _c.cpdp_set_reconcile_staging(self.ctx, stages)

    def set_reconcile_shuffle(self, enable: bool) -> None:
        """True: worker rows split across a warp's lanes, sums by warp shuffles
        (the measured alternative; off by default)."""
        _c.cpdp_set_reconcile_shuffle(self.ctx, enable)

    def reconcile_kernel(self) -> str:
        """The kernel the last reconcile launched ("" before the first)."""
        return _c.cpdp_reconcile_kernel(self.ctx)

    def wait_timeouts(self) -> int:
        """Bounded kernel waits that ran out since the last call (0 expected)."""
        return _c.cpdp_wait_timeouts(self.ctx)

    def set_method(self, method: str) -> None:
        """"cpdp" (default), "localsgd" or "ddp" (the paper's baselines)."""
        _c.cpdp_set_method(self.ctx, _c.METHODS[method])

    def counts(self) -> tuple[int, int]:
        """(gradient means, parameter means) launched so far."""
        return _c.cpdp_get_counts(self.ctx)

    def set_sync_period(self, K: int) -> None:
        _c.cpdp_set_sync_period(self.ctx, K)
        self.K = int(K)

    # -- training-protocol schedule (warmup epochs at K = 1, cosine LR) ----
    def set_schedule(self, steps_per_epoch: int, total_epochs: int, warmup_epochs: int,
                     base_lr: float, min_lr: float = 0.0) -> None:
        _c.cpdp_set_schedule(self.ctx, steps_per_epoch, total_epochs, warmup_epochs, base_lr, min_lr)

    def scheduled_lr(self, epoch: int, t: int) -> float:
        lr = _c.cpdp_scheduled_lr(self.ctx, epoch, t)
        if lr < 0:
            raise ValueError(f"step (epoch={epoch}, t={t}) is outside the schedule")
        return lr

    def is_sync_step_at(self, epoch: int, t: int) -> bool:
        r = _c.cpdp_is_sync_step_at(self.ctx, epoch, t)
        if r < 0:
            raise ValueError(f"step (epoch={epoch}, t={t}) is outside the schedule")
        return bool(r)

    def step_at(self, grads: torch.Tensor, epoch: int, t: int, stream=None) -> bool:
        g = self._grads(grads)
        return _c.cpdp_step_at(self.ctx, g, grad_dtype_code(g), epoch, t, self._stream(stream))

    def close(self) -> None:
        if self.ctx is not None:
            _c.cpdp_destroy(self.ctx)
            self.ctx = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
