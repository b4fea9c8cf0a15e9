"""Feed per-step gradients from page-locked host memory to a CPDPState.

When gradients arrive on the host (the end-to-end setting), the host-to-device
copy of step i+1 can run on a copy engine while the GPU still works on step i.
``HostGradientPipeline`` allocates the two device staging buffers with torch
and hands them to the library (cpdp_bind_staging); each step then goes through
cpdp_step_host / cpdp_step_host_at, which issue the copy on the library's copy
stream and order it against the kernels with events. Argument marshalling only.
"""
from __future__ import annotations

import torch

from . import cpdp as _c
from .state import CPDPState, grad_dtype_code


class HostGradientPipeline:
    def __init__(self, state: CPDPState, dtype: torch.dtype = torch.float32):
        self.state = state
        self.staging = [torch.empty((state.W, state.N), dtype=dtype, device=state.device) for _ in range(2)]
        nbytes = self.staging[0].numel() * self.staging[0].element_size()
        _c.cpdp_bind_staging(state.ctx, self.staging[0], self.staging[1], nbytes)

    def _host(self, host_grads: torch.Tensor) -> torch.Tensor:
        if host_grads.device.type != "cpu" or not host_grads.is_pinned():
            raise ValueError("host gradients must be a page-locked (pinned) CPU tensor")
        st = self.state
        if tuple(host_grads.shape) != (st.W, st.N) or not host_grads.is_contiguous():
            raise ValueError(f"host gradients must be a contiguous ({st.W}, {st.N}) tensor")
        return host_grads

    def step(self, host_grads: torch.Tensor, t: int, steps_per_epoch: int, stream=None) -> bool:
        """cpdp_step on gradients copied from `host_grads` (returns s_t)."""
        g = self._host(host_grads)
        return _c.cpdp_step_host(self.state.ctx, g, grad_dtype_code(g), t, steps_per_epoch,
                                 self.state._stream(stream))

    def step_at(self, host_grads: torch.Tensor, epoch: int, t: int, stream=None) -> bool:
        """cpdp_step_at (the training-protocol schedule) on copied gradients."""
        g = self._host(host_grads)
        return _c.cpdp_step_host_at(self.state.ctx, g, grad_dtype_code(g), epoch, t, self.state._stream(stream))
