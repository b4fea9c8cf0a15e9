"""Python binding of libcpdp (the C ABI declared in include/cpdp.h).

Argument marshalling only: each function has the C entry point's name, turns
Python ints / torch tensors into pointers and sizes, calls the library, and
raises ``CPDPError`` when the status is not CPDP_OK. Every step of the hot path
runs in the library's CUDA kernels; there is no Python or CPU fallback, and a
missing library is an error.
"""
from __future__ import annotations

import ctypes
import os
from pathlib import Path

_LIBRARY = Path(__file__).resolve().parent / "libcpdp.so"

CPDP_OK, CPDP_EINVAL, CPDP_EALIGN, CPDP_ECUDA, CPDP_ESTATE, CPDP_ENOMEM = range(6)
CPDP_F32, CPDP_BF16 = 0, 1
CPDP_METHOD_CPDP, CPDP_METHOD_LOCALSGD, CPDP_METHOD_DDP = 0, 1, 2
METHODS = {"cpdp": CPDP_METHOD_CPDP, "localsgd": CPDP_METHOD_LOCALSGD, "ddp": CPDP_METHOD_DDP}
STATUS_NAMES = {0: "CPDP_OK", 1: "CPDP_EINVAL", 2: "CPDP_EALIGN", 3: "CPDP_ECUDA",
                4: "CPDP_ESTATE", 5: "CPDP_ENOMEM"}

# Every entry point declared in include/cpdp.h.
EXPORTS = ("cpdp_create", "cpdp_bind", "cpdp_init_params", "cpdp_local_step", "cpdp_reconcile",
           "cpdp_is_sync_step", "cpdp_step", "cpdp_set_lr", "cpdp_set_sync_period", "cpdp_set_schedule",
           "cpdp_scheduled_lr", "cpdp_is_sync_step_at", "cpdp_step_at", "cpdp_set_method", "cpdp_get_counts",
           "cpdp_set_adamw", "cpdp_set_optimizer_step", "cpdp_get_optimizer_step", "cpdp_set_state_reconcile",
           "cpdp_set_pdl", "cpdp_bind_staging", "cpdp_step_host", "cpdp_step_host_at",
           "cpdp_step_host_noalloc", "cpdp_bad_index_count", "cpdp_set_reconcile_staging", "cpdp_set_reconcile_shuffle",
           "cpdp_wait_timeouts", "cpdp_reconcile_kernel", "cpdp_withhold_staged_tile", "cpdp_floor_stream", "cpdp_floor_empty",
           "cpdp_floor_columns",
           "cpdp_destroy", "cpdp_last_error")


class CPDPError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


_lib = None


def library_path() -> Path:
    """libcpdp.so in this package, or the library file CPDP_LIBRARY names (e.g.
    the index-checked debug build libcpdp_checked.so)."""
    env = os.environ.get("CPDP_LIBRARY")
    return Path(env) if env else _LIBRARY


def lib() -> ctypes.CDLL:
    """The loaded libcpdp. Raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = library_path()
    if not path.exists():
        raise RuntimeError(f"{path} is not built; run paper_2607_21224_gb300.build.build_library() "
                           "(or __graft_entry__.build()). There is no fallback implementation.")
    L = ctypes.CDLL(str(path))
    vp, i64, c_int, f32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float
    st = c_int
    L.cpdp_create.argtypes = [ctypes.POINTER(vp), c_int, i64, ctypes.POINTER(i64), c_int,
                              f32, f32, f32, c_int, f32, f32]
    L.cpdp_create.restype = st
    L.cpdp_bind.argtypes = [vp, vp, vp, vp, vp]
    L.cpdp_bind.restype = st
    L.cpdp_init_params.argtypes = [vp, vp, vp]
    L.cpdp_init_params.restype = st
    L.cpdp_local_step.argtypes = [vp, vp, c_int, vp]
    L.cpdp_local_step.restype = st
    L.cpdp_reconcile.argtypes = [vp, vp, c_int, vp]
    L.cpdp_reconcile.restype = st
    L.cpdp_is_sync_step.argtypes = [vp, i64, i64]
    L.cpdp_is_sync_step.restype = c_int
    L.cpdp_step.argtypes = [vp, vp, c_int, i64, i64, vp, ctypes.POINTER(c_int)]
    L.cpdp_step.restype = st
    L.cpdp_set_lr.argtypes = [vp, f32]
    L.cpdp_set_lr.restype = st
    L.cpdp_set_sync_period.argtypes = [vp, c_int]
    L.cpdp_set_sync_period.restype = st
    L.cpdp_set_schedule.argtypes = [vp, i64, i64, i64, f32, f32]
    L.cpdp_set_schedule.restype = st
    L.cpdp_scheduled_lr.argtypes = [vp, i64, i64]
    L.cpdp_scheduled_lr.restype = f32
    L.cpdp_is_sync_step_at.argtypes = [vp, i64, i64]
    L.cpdp_is_sync_step_at.restype = c_int
    L.cpdp_step_at.argtypes = [vp, vp, c_int, i64, i64, vp, ctypes.POINTER(c_int)]
    L.cpdp_step_at.restype = st
    L.cpdp_set_method.argtypes = [vp, c_int]
    L.cpdp_set_method.restype = st
    L.cpdp_get_counts.argtypes = [vp, ctypes.POINTER(i64), ctypes.POINTER(i64)]
    L.cpdp_get_counts.restype = st
    L.cpdp_set_adamw.argtypes = [vp, f32, f32, f32, vp]
    L.cpdp_set_adamw.restype = st
    L.cpdp_set_state_reconcile.argtypes = [vp, c_int]
    L.cpdp_set_state_reconcile.restype = st
    L.cpdp_set_pdl.argtypes = [vp, c_int]
    L.cpdp_set_pdl.restype = st
    L.cpdp_set_optimizer_step.argtypes = [vp, i64]
    L.cpdp_set_optimizer_step.restype = st
    L.cpdp_get_optimizer_step.argtypes = [vp, ctypes.POINTER(i64)]
    L.cpdp_get_optimizer_step.restype = st
    L.cpdp_bind_staging.argtypes = [vp, vp, vp, ctypes.c_size_t]
    L.cpdp_bind_staging.restype = st
    L.cpdp_step_host.argtypes = [vp, vp, c_int, i64, i64, vp, ctypes.POINTER(c_int)]
    L.cpdp_step_host.restype = st
    L.cpdp_step_host_at.argtypes = [vp, vp, c_int, i64, i64, vp, ctypes.POINTER(c_int)]
    L.cpdp_step_host_at.restype = st
    L.cpdp_step_host_noalloc.argtypes = [vp, vp, c_int, i64, i64, vp, ctypes.POINTER(c_int)]
    L.cpdp_step_host_noalloc.restype = st
    L.cpdp_bad_index_count.argtypes = [vp, ctypes.POINTER(i64)]
    L.cpdp_bad_index_count.restype = st
    L.cpdp_set_reconcile_staging.argtypes = [vp, c_int]
    L.cpdp_set_reconcile_staging.restype = st
    L.cpdp_set_reconcile_shuffle.argtypes = [vp, c_int]
    L.cpdp_set_reconcile_shuffle.restype = st
    L.cpdp_withhold_staged_tile.argtypes = [vp, i64]
    L.cpdp_withhold_staged_tile.restype = st
    L.cpdp_wait_timeouts.argtypes = [vp, ctypes.POINTER(i64)]
    L.cpdp_wait_timeouts.restype = st
    L.cpdp_reconcile_kernel.argtypes = [vp, ctypes.POINTER(ctypes.c_char_p)]
    L.cpdp_reconcile_kernel.restype = st
    L.cpdp_floor_stream.argtypes = [ctypes.POINTER(vp), c_int, ctypes.POINTER(vp), c_int, ctypes.POINTER(vp), c_int, i64,
                                    ctypes.c_uint, vp]
    L.cpdp_floor_stream.restype = st
    L.cpdp_floor_empty.argtypes = [ctypes.c_uint, vp]
    L.cpdp_floor_empty.restype = st
    L.cpdp_floor_columns.argtypes = [vp, vp, vp, vp, c_int, vp, vp, c_int, i64, c_int, c_int, vp]
    L.cpdp_floor_columns.restype = st
    L.cpdp_destroy.argtypes = [vp]
    L.cpdp_destroy.restype = st
    L.cpdp_last_error.argtypes = [vp]
    L.cpdp_last_error.restype = ctypes.c_char_p
    _lib = L
    return L


def _check(status: int, ctx=None) -> None:
    if status != CPDP_OK:
        raise CPDPError(status, cpdp_last_error(ctx))


def _addr(x) -> int | None:
    """A raw address from an int, None, or a tensor-like with data_ptr()."""
    if x is None or isinstance(x, int):
        return x
    return x.data_ptr()


def cpdp_last_error(ctx=None) -> str:
    msg = lib().cpdp_last_error(ctx)
    return msg.decode() if msg else ""


def cpdp_create(W: int, N: int, tensor_offsets, lr: float, momentum: float, weight_decay: float,
                K: int, slowmo_beta: float, slowmo_alpha: float = 1.0) -> int:
    """Returns the context handle (an int). tensor_offsets: sequence of
    num_tensors+1 prefix offsets, or None for one tensor of N elements."""
    out = ctypes.c_void_p()
    if tensor_offsets is None:
        offs, n_t = None, 0
    else:
        vals = [int(x) for x in tensor_offsets]
        offs, n_t = (ctypes.c_int64 * len(vals))(*vals), len(vals) - 1
    _check(lib().cpdp_create(ctypes.byref(out), int(W), int(N), offs, n_t, float(lr), float(momentum),
                             float(weight_decay), int(K), float(slowmo_beta), float(slowmo_alpha)))
    return out.value


def cpdp_bind(ctx: int, params, mom, anchor, slow_v) -> None:
    _check(lib().cpdp_bind(ctx, _addr(params), _addr(mom), _addr(anchor), _addr(slow_v)), ctx)


def cpdp_init_params(ctx: int, theta0, stream: int | None = None) -> None:
    _check(lib().cpdp_init_params(ctx, _addr(theta0), stream), ctx)


def cpdp_local_step(ctx: int, grads, dtype: int, stream: int | None = None) -> None:
    _check(lib().cpdp_local_step(ctx, _addr(grads), int(dtype), stream), ctx)


def cpdp_reconcile(ctx: int, grads, dtype: int, stream: int | None = None) -> None:
    _check(lib().cpdp_reconcile(ctx, _addr(grads), int(dtype), stream), ctx)


def cpdp_is_sync_step(ctx: int, t: int, steps_per_epoch: int) -> int:
    return lib().cpdp_is_sync_step(ctx, int(t), int(steps_per_epoch))


def cpdp_step(ctx: int, grads, dtype: int, t: int, steps_per_epoch: int, stream: int | None = None) -> bool:
    did = ctypes.c_int(-1)
    _check(lib().cpdp_step(ctx, _addr(grads), int(dtype), int(t), int(steps_per_epoch), stream,
                           ctypes.byref(did)), ctx)
    return bool(did.value)


def cpdp_set_lr(ctx: int, lr: float) -> None:
    _check(lib().cpdp_set_lr(ctx, float(lr)), ctx)


def cpdp_set_sync_period(ctx: int, K: int) -> None:
    _check(lib().cpdp_set_sync_period(ctx, int(K)), ctx)


def cpdp_set_schedule(ctx: int, steps_per_epoch: int, total_epochs: int, warmup_epochs: int,
                      base_lr: float, min_lr: float = 0.0) -> None:
    _check(lib().cpdp_set_schedule(ctx, int(steps_per_epoch), int(total_epochs), int(warmup_epochs),
                                   float(base_lr), float(min_lr)), ctx)


def cpdp_scheduled_lr(ctx: int, epoch: int, t: int) -> float:
    return float(lib().cpdp_scheduled_lr(ctx, int(epoch), int(t)))


def cpdp_is_sync_step_at(ctx: int, epoch: int, t: int) -> int:
    return lib().cpdp_is_sync_step_at(ctx, int(epoch), int(t))


def cpdp_step_at(ctx: int, grads, dtype: int, epoch: int, t: int, stream: int | None = None) -> bool:
    did = ctypes.c_int(-1)
    _check(lib().cpdp_step_at(ctx, _addr(grads), int(dtype), int(epoch), int(t), stream, ctypes.byref(did)), ctx)
    return bool(did.value)


def cpdp_set_method(ctx: int, method: int) -> None:
    _check(lib().cpdp_set_method(ctx, int(method)), ctx)


def cpdp_get_counts(ctx: int) -> tuple[int, int]:
    g, p = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().cpdp_get_counts(ctx, ctypes.byref(g), ctypes.byref(p)), ctx)
    return g.value, p.value


def cpdp_set_adamw(ctx: int, beta1: float, beta2: float, eps: float, exp_avg_sq) -> None:
    _check(lib().cpdp_set_adamw(ctx, float(beta1), float(beta2), float(eps), _addr(exp_avg_sq)), ctx)


def cpdp_set_state_reconcile(ctx: int, enable: bool) -> None:
    _check(lib().cpdp_set_state_reconcile(ctx, 1 if enable else 0), ctx)


def cpdp_set_pdl(ctx: int, enable: bool) -> None:
    _check(lib().cpdp_set_pdl(ctx, 1 if enable else 0), ctx)


def cpdp_set_optimizer_step(ctx: int, step: int) -> None:
    _check(lib().cpdp_set_optimizer_step(ctx, int(step)), ctx)


def cpdp_get_optimizer_step(ctx: int) -> int:
    v = ctypes.c_int64()
    _check(lib().cpdp_get_optimizer_step(ctx, ctypes.byref(v)), ctx)
    return v.value


def cpdp_bind_staging(ctx: int, stage0, stage1, bytes_each: int) -> None:
    _check(lib().cpdp_bind_staging(ctx, _addr(stage0), _addr(stage1), int(bytes_each)), ctx)


def cpdp_step_host(ctx: int, host_grads, dtype: int, t: int, steps_per_epoch: int,
                   stream: int | None = None) -> bool:
    did = ctypes.c_int(-1)
    _check(lib().cpdp_step_host(ctx, _addr(host_grads), int(dtype), int(t), int(steps_per_epoch), stream,
                                ctypes.byref(did)), ctx)
    return bool(did.value)


def cpdp_step_host_at(ctx: int, host_grads, dtype: int, epoch: int, t: int, stream: int | None = None) -> bool:
    did = ctypes.c_int(-1)
    _check(lib().cpdp_step_host_at(ctx, _addr(host_grads), int(dtype), int(epoch), int(t), stream,
                                   ctypes.byref(did)), ctx)
    return bool(did.value)


# Size of the staging area built into the library (CPDP_NOALLOC_STAGING_BYTES).
CPDP_NOALLOC_STAGING_BYTES = 64 << 20


def cpdp_step_host_noalloc(ctx: int, host_grads, dtype: int, t: int, steps_per_epoch: int,
                           stream: int | None = None) -> bool:
    """cpdp_step_host through the library's built-in staging area: for callers
    that cannot allocate device staging buffers (returns s_t)."""
    did = ctypes.c_int(-1)
    _check(lib().cpdp_step_host_noalloc(ctx, _addr(host_grads), int(dtype), int(t), int(steps_per_epoch), stream,
                                        ctypes.byref(did)), ctx)
    return bool(did.value)


def cpdp_bad_index_count(ctx: int) -> int:
    """Out-of-range kernel indices counted since the last call on ctx's device
    (the index-checked debug build; -1 from a release build)."""
    v = ctypes.c_int64()
    _check(lib().cpdp_bad_index_count(ctx, ctypes.byref(v)), ctx)
    return v.value


def cpdp_set_reconcile_staging(ctx: int, stages: int) -> None:
    """0: the reconcile loads its rows directly (default); 2..8: rows staged
    through a ring of that many shared-memory slots by bulk copies."""
    _check(lib().cpdp_set_reconcile_staging(ctx, int(stages)), ctx)


def cpdp_set_reconcile_shuffle(ctx: int, enable: bool) -> None:
    """True: the reconcile splits the worker rows across a warp's lanes and adds
    the partial sums with warp shuffles (the measured alternative)."""
    _check(lib().cpdp_set_reconcile_shuffle(ctx, 1 if enable else 0), ctx)


def cpdp_withhold_staged_tile(ctx: int, tile: int) -> None:
    """Test of the bounded waits: the next staged reconcile leaves out the
    loads of column tile `tile`, and its waits for it run out."""
    _check(lib().cpdp_withhold_staged_tile(ctx, int(tile)), ctx)


def cpdp_reconcile_kernel(ctx: int) -> str:
    """The name of the kernel the last reconcile on ctx launched ("" before
    the first)."""
    v = ctypes.c_char_p()
    _check(lib().cpdp_reconcile_kernel(ctx, ctypes.byref(v)), ctx)
    return v.value.decode() if v.value else ""


def cpdp_wait_timeouts(ctx: int) -> int:
    """Bounded kernel waits that ran out since the last call on ctx's device."""
    v = ctypes.c_int64()
    _check(lib().cpdp_wait_timeouts(ctx, ctypes.byref(v)), ctx)
    return v.value


class FloorRows:
    """The row pointers of one floor launch, marshalled once so that repeated
    launches (a timed loop) spend no host time rebuilding them."""

    def __init__(self, inputs, outputs, inputs_bf16=()):
        self.n_in, self.n_in_bf16, self.n_out = len(inputs), len(inputs_bf16), len(outputs)
        self.ins = (ctypes.c_void_p * max(1, self.n_in))(*[_addr(x) for x in inputs])
        self.ins_bf16 = (ctypes.c_void_p * max(1, self.n_in_bf16))(*[_addr(x) for x in inputs_bf16])
        self.outs = (ctypes.c_void_p * max(1, self.n_out))(*[_addr(x) for x in outputs])


def cpdp_floor_stream(inputs, outputs=None, n: int = 0, grid: int = 0, stream: int | None = None,
                      inputs_bf16=()) -> None:
    """One launch of the plain streaming floor kernel over `inputs` (float32
    rows), `inputs_bf16` (bf16 rows) and `outputs` (float32 rows), n elements
    each (tensors or addresses), or over the rows of a FloorRows passed as
    `inputs`."""
    rows = inputs if isinstance(inputs, FloorRows) else FloorRows(inputs, outputs, inputs_bf16)
    _check(lib().cpdp_floor_stream(rows.ins, rows.n_in, rows.ins_bf16, rows.n_in_bf16, rows.outs, rows.n_out, int(n),
                                   int(grid), stream))


def cpdp_floor_empty(grid: int = 0, stream: int | None = None) -> None:
    """One launch of the empty floor kernel."""
    _check(lib().cpdp_floor_empty(int(grid), stream))


def cpdp_floor_columns(params, mom, sq, grads, grad_dtype: int, anchor, slow_v, W: int, N: int, chunk_rows: int,
                       blocks_per_sm: int, stream: int | None = None) -> None:
    """One launch of the column-walk floor kernel over a reconcile's arrays
    (tensors or addresses; sq may be None)."""
    _check(lib().cpdp_floor_columns(_addr(params), _addr(mom), None if sq is None else _addr(sq), _addr(grads),
                                    int(grad_dtype), _addr(anchor), _addr(slow_v), int(W), int(N), int(chunk_rows),
                                    int(blocks_per_sm), stream))


def cpdp_destroy(ctx: int | None) -> None:
    _check(lib().cpdp_destroy(ctx))
