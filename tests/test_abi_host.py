"""Host-side tests of libcpdp's C ABI that need no GPU: the library loads,
exports every entry point include/cpdp.h declares, validates its arguments,
and implements the synchronization schedule exactly like the oracle."""
import ctypes
import math
import re
from pathlib import Path

import pytest

from paper_2607_21224_gb300 import build, cpdp
from paper_2607_21224_gb300.cpdp import CPDPError

HEADER = Path(__file__).resolve().parents[1] / "include" / "cpdp.h"
GOOD = dict(W=4, N=100, tensor_offsets=[0, 40, 100], lr=0.1, momentum=0.9, weight_decay=5e-4,
            K=4, slowmo_beta=0.5, slowmo_alpha=1.0)


@pytest.fixture(scope="module")
def L():
    build.build_library()
    return cpdp.lib()


def declared_functions() -> set[str]:
    text = HEADER.read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return set(re.findall(r"\b(cpdp_[a-z_]+)\s*\(", text))


def test_header_and_binding_agree():
    assert declared_functions() == set(cpdp.EXPORTS)


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name
        assert ctypes.cast(getattr(L, name), ctypes.c_void_p).value


def test_library_is_in_tree(L):
    assert cpdp.library_path().parent == Path(cpdp.__file__).resolve().parent
    assert cpdp.library_path().exists()


def test_create_destroy_roundtrip(L):
    ctx = cpdp.cpdp_create(**GOOD)
    assert ctx
    assert cpdp.cpdp_last_error(ctx) == ""
    cpdp.cpdp_destroy(ctx)


@pytest.mark.parametrize("bad", [
    dict(W=0), dict(W=4097), dict(N=0), dict(N=-5), dict(lr=0.0), dict(lr=-1.0),
    dict(lr=float("nan")), dict(momentum=-0.1), dict(weight_decay=-1e-4), dict(K=0),
    dict(slowmo_beta=1.0), dict(slowmo_beta=-0.1), dict(slowmo_beta=float("inf")),
    dict(slowmo_alpha=0.0), dict(tensor_offsets=[1, 100]), dict(tensor_offsets=[0, 50, 50, 100]),
    dict(tensor_offsets=[0, 99]), dict(tensor_offsets=[0, 60, 40, 100]),
])
def test_create_rejects_invalid_arguments(L, bad):
    args = {**GOOD, **bad}
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_create(**args)
    assert e.value.status == cpdp.CPDP_EINVAL
    assert cpdp.cpdp_last_error(None)  # message recorded for the calling thread


def test_create_null_out_pointer(L):
    assert L.cpdp_create(None, 1, 4, None, 0, 0.1, 0.9, 0.0, 1, 0.5, 1.0) == cpdp.CPDP_EINVAL


def test_offsets_optional(L):
    ctx = cpdp.cpdp_create(**{**GOOD, "tensor_offsets": None})
    cpdp.cpdp_destroy(ctx)


def test_double_destroy_and_null(L):
    ctx = cpdp.cpdp_create(**GOOD)
    cpdp.cpdp_destroy(ctx)
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_destroy(ctx)
    assert e.value.status == cpdp.CPDP_EINVAL
    cpdp.cpdp_destroy(None)  # NULL is accepted
    assert L.cpdp_destroy(None) == cpdp.CPDP_OK


def test_calls_on_dead_or_null_context(L):
    ctx = cpdp.cpdp_create(**GOOD)
    cpdp.cpdp_destroy(ctx)
    assert L.cpdp_set_lr(ctx, ctypes.c_float(0.2)) == cpdp.CPDP_EINVAL
    assert L.cpdp_is_sync_step(ctx, 1, 4) == -1
    assert L.cpdp_local_step(None, None, 0, None) == cpdp.CPDP_EINVAL
    assert L.cpdp_reconcile(None, None, 0, None) == cpdp.CPDP_EINVAL
    assert cpdp.cpdp_last_error(ctx) == "not a live context"


def test_steps_before_bind_are_state_errors(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        for fn in (cpdp.cpdp_local_step, cpdp.cpdp_reconcile):
            with pytest.raises(CPDPError) as e:
                fn(ctx, 1 << 20, cpdp.CPDP_F32)
            assert e.value.status == cpdp.CPDP_ESTATE
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_init_params(ctx, 1 << 20)
        assert e.value.status == cpdp.CPDP_ESTATE
    finally:
        cpdp.cpdp_destroy(ctx)


def test_bind_validates_before_touching_cuda(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        base = 1 << 32
        sb, rb = 4 * 100 * 4, 100 * 4
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_bind(ctx, 0, base + sb, base + 2 * sb, base + 2 * sb + rb)
        assert e.value.status == cpdp.CPDP_EINVAL
        with pytest.raises(CPDPError) as e:  # misaligned
            cpdp.cpdp_bind(ctx, base + 4, base + sb + 16, base + 2 * sb + 32, base + 2 * sb + rb + 32)
        assert e.value.status == cpdp.CPDP_EALIGN
        with pytest.raises(CPDPError) as e:  # params and mom overlap
            cpdp.cpdp_bind(ctx, base, base + sb - 16, base + 4 * sb, base + 5 * sb)
        assert e.value.status == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_set_lr(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        cpdp.cpdp_set_lr(ctx, 0.05)
        for bad in (0.0, -1.0, float("nan"), float("inf")):
            with pytest.raises(CPDPError):
                cpdp.cpdp_set_lr(ctx, bad)
    finally:
        cpdp.cpdp_destroy(ctx)


def test_schedule_matches_oracle_and_table2(L, oracle_lib):
    """cpdp_is_sync_step against the oracle's eq. 4 + epoch-end rule, and the
    ceil(T/K) reconciles per epoch of Table 2, bit-exact over a grid of T, K."""
    for K in range(1, 11):
        ctx = cpdp.cpdp_create(**{**GOOD, "K": K})
        try:
            for T in range(1, 34):
                got = [cpdp.cpdp_is_sync_step(ctx, t, T) for t in range(1, T + 1)]
                want = [int(oracle_lib.is_sync_step(t, K, T)) for t in range(1, T + 1)]
                assert got == want, (K, T)
                assert sum(got) == math.ceil(T / K)
            assert cpdp.cpdp_is_sync_step(ctx, 0, 5) == -1
            assert cpdp.cpdp_is_sync_step(ctx, 6, 5) == -1
        finally:
            cpdp.cpdp_destroy(ctx)


def test_step_rejects_out_of_range_t(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_step(ctx, 1 << 20, cpdp.CPDP_F32, 0, 4)
        assert e.value.status == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(cpdp, "_lib", None)
    monkeypatch.setattr(cpdp, "_LIBRARY", tmp_path / "libcpdp.so")
    with pytest.raises(RuntimeError, match="not built"):
        cpdp.lib()


# ---------------------------------------------------------------------------
# training-protocol schedule (host-only entry points)
# ---------------------------------------------------------------------------
def test_scheduled_lr_matches_oracle(L, oracle_lib):
    """cpdp_scheduled_lr equals the oracle's double-precision schedule rounded
    to float32, at every step of several schedules."""
    import numpy as np
    for T, E, We, base, lo in ((7, 6, 2, 0.4, 0.0), (16, 3, 1, 0.1, 1e-3), (5, 4, 0, 5e-4, 0.0)):
        ctx = cpdp.cpdp_create(**GOOD)
        try:
            cpdp.cpdp_set_schedule(ctx, T, E, We, base, lo)
            b32, l32 = float(np.float32(base)), float(np.float32(lo))
            for e in range(E):
                for t in range(1, T + 1):
                    want = float(np.float32(oracle_lib.scheduled_lr(b32, l32, We * T, E * T, e * T + t - 1)))
                    assert cpdp.cpdp_scheduled_lr(ctx, e, t) == want, (e, t)
            assert cpdp.cpdp_scheduled_lr(ctx, E, 1) == -1.0
            assert cpdp.cpdp_scheduled_lr(ctx, 0, T + 1) == -1.0
        finally:
            cpdp.cpdp_destroy(ctx)


def test_sync_at_matches_oracle(L, oracle_lib):
    for K, T, E, We in ((2, 7, 5, 2), (4, 16, 3, 1), (8, 5, 3, 0), (1, 4, 2, 1)):
        ctx = cpdp.cpdp_create(**{**GOOD, "K": K})
        try:
            cpdp.cpdp_set_schedule(ctx, T, E, We, 0.1, 0.0)
            for e in range(E):
                for t in range(1, T + 1):
                    assert cpdp.cpdp_is_sync_step_at(ctx, e, t) == int(oracle_lib.is_sync_step_at(e, t, K, T, We))
            assert cpdp.cpdp_is_sync_step_at(ctx, -1, 1) == -1
        finally:
            cpdp.cpdp_destroy(ctx)


@pytest.mark.parametrize("bad", [(0, 5, 1, 0.1, 0.0), (4, 0, 0, 0.1, 0.0), (4, 5, 5, 0.1, 0.0),
                                 (4, 5, -1, 0.1, 0.0), (4, 5, 1, 0.0, 0.0), (4, 5, 1, 0.1, 0.2),
                                 (4, 5, 1, 0.1, -0.1), (4, 5, 1, float("nan"), 0.0)])
def test_set_schedule_validation(L, bad):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_set_schedule(ctx, *bad)
        assert e.value.status == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_step_at_needs_schedule_and_range(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_step_at(ctx, 1 << 20, cpdp.CPDP_F32, 0, 1)
        assert e.value.status == cpdp.CPDP_ESTATE
        assert cpdp.cpdp_is_sync_step_at(ctx, 0, 1) == -1
        cpdp.cpdp_set_schedule(ctx, 4, 2, 1, 0.1)
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_step_at(ctx, 1 << 20, cpdp.CPDP_F32, 2, 1)
        assert e.value.status == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_set_sync_period(L):
    ctx = cpdp.cpdp_create(**{**GOOD, "K": 4})
    try:
        assert [cpdp.cpdp_is_sync_step(ctx, t, 8) for t in range(1, 9)] == [0, 0, 0, 1, 0, 0, 0, 1]
        cpdp.cpdp_set_sync_period(ctx, 1)
        assert all(cpdp.cpdp_is_sync_step(ctx, t, 8) == 1 for t in range(1, 9))
        with pytest.raises(CPDPError):
            cpdp.cpdp_set_sync_period(ctx, 0)
    finally:
        cpdp.cpdp_destroy(ctx)


def test_set_method_and_counts(L):
    ctx = cpdp.cpdp_create(**{**GOOD, "K": 3})
    try:
        assert cpdp.cpdp_get_counts(ctx) == (0, 0)
        cpdp.cpdp_set_method(ctx, cpdp.CPDP_METHOD_DDP)
        assert all(cpdp.cpdp_is_sync_step(ctx, t, 7) == 1 for t in range(1, 8))
        cpdp.cpdp_set_method(ctx, cpdp.CPDP_METHOD_LOCALSGD)
        assert [cpdp.cpdp_is_sync_step(ctx, t, 7) for t in range(1, 8)] == [0, 0, 1, 0, 0, 1, 1]
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_set_method(ctx, 3)
        assert e.value.status == cpdp.CPDP_EINVAL
        assert L.cpdp_get_counts(ctx, None, None) == cpdp.CPDP_OK
    finally:
        cpdp.cpdp_destroy(ctx)


def test_adamw_needs_bound_state_and_step_counter(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_set_adamw(ctx, 0.9, 0.999, 1e-8, 1 << 20)
        assert e.value.status == cpdp.CPDP_ESTATE
        assert cpdp.cpdp_get_optimizer_step(ctx) == 0
        cpdp.cpdp_set_optimizer_step(ctx, 17)
        assert cpdp.cpdp_get_optimizer_step(ctx) == 17
        with pytest.raises(CPDPError):
            cpdp.cpdp_set_optimizer_step(ctx, -1)
    finally:
        cpdp.cpdp_destroy(ctx)


def test_set_state_reconcile(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        cpdp.cpdp_set_state_reconcile(ctx, True)
        cpdp.cpdp_set_state_reconcile(ctx, False)
        assert L.cpdp_set_state_reconcile(ctx, 2) == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_set_pdl(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        cpdp.cpdp_set_pdl(ctx, False)
        cpdp.cpdp_set_pdl(ctx, True)
        assert L.cpdp_set_pdl(ctx, 2) == cpdp.CPDP_EINVAL
        assert L.cpdp_set_pdl(None, 1) == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_host_staging_needs_binding(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_bind_staging(ctx, 1 << 20, 1 << 21, 4096)
        assert e.value.status == cpdp.CPDP_ESTATE
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_step_host(ctx, 1 << 20, cpdp.CPDP_F32, 1, 4)
        assert e.value.status == cpdp.CPDP_ESTATE
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_step_host(ctx, 1 << 20, cpdp.CPDP_F32, 9, 4)
        assert e.value.status == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_bad_index_count_is_minus_one_in_a_release_build(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        assert cpdp.cpdp_bad_index_count(ctx) == -1
        assert L.cpdp_bad_index_count(ctx, None) == cpdp.CPDP_EINVAL
        assert L.cpdp_bad_index_count(None, None) == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)


def test_floor_stream_validates_before_launching(L):
    """The floor kernel's arguments are checked on the host; nothing is
    launched on a bad call (so these run without a GPU)."""
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_floor_stream([], [], 16)
    assert e.value.status == cpdp.CPDP_EINVAL
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_floor_stream([16] * 129, [], 16)
    assert e.value.status == cpdp.CPDP_EINVAL
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_floor_stream([16], [32], 6)
    assert e.value.status == cpdp.CPDP_EINVAL and "multiple of 4" in str(e.value)
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_floor_stream([24], [32], 16)
    assert e.value.status == cpdp.CPDP_EALIGN
    # bf16 input rows: 8-byte aligned, at most 128
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_floor_stream([], [32], 16, inputs_bf16=[20])
    assert e.value.status == cpdp.CPDP_EALIGN and "bf16 input row 0" in str(e.value)
    with pytest.raises(CPDPError) as e:
        cpdp.cpdp_floor_stream([16], [32], 16, inputs_bf16=[8] * 129)
    assert e.value.status == cpdp.CPDP_EINVAL


def test_floor_columns_validates_before_launching(L):
    """The column-walk floor's arguments are checked on the host; nothing is
    launched on a bad call (so these run without a GPU)."""
    ok = dict(params=16, mom=32, sq=None, grads=48, grad_dtype=cpdp.CPDP_F32, anchor=64, slow_v=80, W=2, N=8,
              chunk_rows=2, blocks_per_sm=4)
    bad = [(dict(W=0), cpdp.CPDP_EINVAL), (dict(W=4097), cpdp.CPDP_EINVAL), (dict(N=6), cpdp.CPDP_EINVAL),
           (dict(N=0), cpdp.CPDP_EINVAL), (dict(grad_dtype=7), cpdp.CPDP_EINVAL),
           (dict(chunk_rows=4, blocks_per_sm=3), cpdp.CPDP_EINVAL), (dict(chunk_rows=1, blocks_per_sm=4), cpdp.CPDP_EINVAL),
           (dict(params=None), cpdp.CPDP_EALIGN), (dict(mom=40), cpdp.CPDP_EALIGN), (dict(sq=24), cpdp.CPDP_EALIGN),
           (dict(grads=40), cpdp.CPDP_EALIGN), (dict(grads=44, grad_dtype=cpdp.CPDP_BF16), cpdp.CPDP_EALIGN),
           (dict(anchor=None), cpdp.CPDP_EALIGN)]
    for change, status in bad:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_floor_columns(**{**ok, **change})
        assert e.value.status == status, change


def test_staging_and_timeouts_need_bound_state(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_set_reconcile_staging(ctx, 2)
        assert e.value.status == cpdp.CPDP_ESTATE
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_wait_timeouts(ctx)
        assert e.value.status == cpdp.CPDP_ESTATE
    finally:
        cpdp.cpdp_destroy(ctx)


def test_reconcile_kernel_before_any_reconcile(L):
    """Host-only: "" until a reconcile has run; invalid context or NULL name
    refused without touching the output."""
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        assert cpdp.cpdp_reconcile_kernel(ctx) == ""
        assert L.cpdp_reconcile_kernel(ctx, None) == cpdp.CPDP_EINVAL
    finally:
        cpdp.cpdp_destroy(ctx)
    name = ctypes.c_char_p(b"kept")
    assert L.cpdp_reconcile_kernel(None, ctypes.byref(name)) == cpdp.CPDP_EINVAL
    assert name.value == b"kept"


def test_withhold_needs_the_staged_reconcile(L):
    ctx = cpdp.cpdp_create(**GOOD)
    try:
        with pytest.raises(CPDPError) as e:
            cpdp.cpdp_withhold_staged_tile(ctx, 0)
        assert e.value.status == cpdp.CPDP_ESTATE
    finally:
        cpdp.cpdp_destroy(ctx)
