"""Feed per-step gradients from page-locked host memory to a CPDPState.

When gradients arrive on the host (the end-to-end setting), the host-to-device
copy of step i+1 can run on a copy engine while the GPU still works on step i.
``HostGradientPipeline`` does that with a dedicated copy stream and a ring of
`depth` device buffers: a buffer is refilled only after the step that read it
has finished (an event recorded on the compute stream), and a step starts only
after its buffer's copy has landed (an event recorded on the copy stream).
Torch provides the streams, events and copies; every step of the method still
runs in libcpdp's kernels.
"""
from __future__ import annotations

import torch

from .state import CPDPState


class HostGradientPipeline:
    def __init__(self, state: CPDPState, dtype: torch.dtype = torch.float32, depth: int = 2):
        if depth < 1:
            raise ValueError("depth must be >= 1")
        self.state = state
        dev = state.device
        self.copy_stream = torch.cuda.Stream(dev)
        self.buffers = [torch.empty((state.W, state.N), dtype=dtype, device=dev) for _ in range(depth)]
        self.copied = [torch.cuda.Event() for _ in range(depth)]
        self.consumed = [torch.cuda.Event() for _ in range(depth)]
        self.in_use = [False] * depth
        self.count = 0

    def _stage(self, host_grads: torch.Tensor) -> torch.Tensor:
        if host_grads.device.type != "cpu" or not host_grads.is_pinned():
            raise ValueError("host gradients must be a page-locked (pinned) CPU tensor")
        k = self.count % len(self.buffers)
        buf = self.buffers[k]
        if buf.shape != host_grads.shape or buf.dtype != host_grads.dtype:
            raise ValueError(f"expected {tuple(buf.shape)} {buf.dtype}, got {tuple(host_grads.shape)} "
                             f"{host_grads.dtype}")
        if self.in_use[k]:
            self.copy_stream.wait_event(self.consumed[k])
        with torch.cuda.stream(self.copy_stream):
            buf.copy_(host_grads, non_blocking=True)
            self.copied[k].record(self.copy_stream)
        return buf

    def _finish(self, stream: torch.cuda.Stream) -> None:
        k = self.count % len(self.buffers)
        self.consumed[k].record(stream)
        self.in_use[k] = True
        self.count += 1

    def _compute_stream(self, stream) -> torch.cuda.Stream:
        return torch.cuda.current_stream(self.state.device) if stream is None else stream

    def step(self, host_grads: torch.Tensor, t: int, steps_per_epoch: int, stream=None) -> bool:
        """cpdp_step on gradients copied from `host_grads` (returns s_t)."""
        stream = self._compute_stream(stream)
        buf = self._stage(host_grads)
        stream.wait_event(self.copied[self.count % len(self.buffers)])
        synced = self.state.step(buf, t, steps_per_epoch, stream=stream)
        self._finish(stream)
        return synced

    def step_at(self, host_grads: torch.Tensor, epoch: int, t: int, stream=None) -> bool:
        """cpdp_step_at (the training-protocol schedule) on copied gradients."""
        stream = self._compute_stream(stream)
        buf = self._stage(host_grads)
        stream.wait_event(self.copied[self.count % len(self.buffers)])
        synced = self.state.step_at(buf, epoch, t, stream=stream)
        self._finish(stream)
        return synced
