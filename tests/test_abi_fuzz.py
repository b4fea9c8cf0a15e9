"""Property-based checks of the C ABI's host-side logic (no GPU): argument
validation of cpdp_create against the rules include/cpdp.h states, the
synchronization indicator against eq. 4 with the epoch-end rule of Sec. 3.1,
and the training-protocol schedule against the oracle. Where hypothesis is
not installed, tests/conftest.py leaves this module out of collection."""
import ctypes
import math

import numpy as np
import pytest

from paper_2607_21224_gb300 import cpdp

from hypothesis import given, settings, strategies as st

SPECIAL = [0.0, -0.0, 1.0, -1.0, 0.5, 0.999, 1.0 - 2 ** -24, 1e-30, float("nan"), float("inf"), float("-inf")]
floats = st.one_of(st.sampled_from(SPECIAL), st.floats(min_value=-1e30, max_value=1e30, allow_nan=False))


def f32(x: float) -> float:
    return float(np.float32(x))


@st.composite
def offsets_for(draw, N: int):
    kind = draw(st.sampled_from(["none", "valid", "bad_start", "not_increasing", "bad_end", "negative_count"]))
    if kind == "none" or N < 1:
        return kind, None, 0
    k = draw(st.integers(min_value=1, max_value=min(8, N)))
    cuts = sorted(draw(st.sets(st.integers(min_value=1, max_value=N - 1), max_size=k - 1))) if N > 1 else []
    offs = [0, *cuts, N]
    if kind == "bad_start":
        offs[0] = 1
    elif kind == "not_increasing" and len(offs) > 2:
        offs[1] = offs[2]
    elif kind == "bad_end":
        offs[-1] = N + 1
    elif kind == "negative_count":
        return kind, offs, -1
    return kind, offs, len(offs) - 1


def expected_ok(W, N, kind, offs, count, lr, mu, wd, K, beta, alpha) -> bool:
    if not (1 <= W <= 4096) or N < 1 or N > (1 << 40) // W:
        return False
    hyper = [f32(x) for x in (lr, mu, wd, beta, alpha)]
    if not all(math.isfinite(x) for x in hyper):
        return False
    lr, mu, wd, beta, alpha = hyper
    if not (lr > 0 and mu >= 0 and wd >= 0 and K >= 1 and 0 <= beta < 1 and alpha > 0):
        return False
    if count < 0:
        return False
    if count > 0:
        return offs[0] == 0 and all(b > a for a, b in zip(offs, offs[1:])) and offs[-1] == N
    return True


@settings(max_examples=400, deadline=None)
@given(W=st.one_of(st.integers(-2, 8), st.sampled_from([4095, 4096, 4097])),
       N=st.one_of(st.integers(-2, 1000), st.sampled_from([1 << 36, (1 << 38) + 1])),
       lr=floats, mu=floats, wd=floats, K=st.integers(-2, 20), beta=floats, alpha=floats, data=st.data())
def test_create_accepts_exactly_the_documented_arguments(W, N, lr, mu, wd, K, beta, alpha, data):
    L = cpdp.lib()
    kind, offs, count = data.draw(offsets_for(N))
    arr = (ctypes.c_int64 * len(offs))(*offs) if offs else None
    out = ctypes.c_void_p()
    status = L.cpdp_create(ctypes.byref(out), W, N, arr, count, lr, mu, wd, K, beta, alpha)
    want = expected_ok(W, N, kind, offs, count, lr, mu, wd, K, beta, alpha)
    assert (status == cpdp.CPDP_OK) == want, (status, W, N, kind, offs, count, lr, mu, wd, K, beta, alpha)
    if status == cpdp.CPDP_OK:
        assert out.value is not None
        assert L.cpdp_destroy(out) == cpdp.CPDP_OK
    else:
        assert status == cpdp.CPDP_EINVAL and out.value is None
        assert cpdp.cpdp_last_error(None)


@settings(max_examples=200, deadline=None)
@given(K=st.integers(1, 40), T=st.integers(1, 200), method=st.sampled_from(["cpdp", "localsgd", "ddp"]),
       t=st.integers(-3, 210))
def test_sync_indicator_is_eq4_with_the_epoch_end_rule(K, T, method, t):
    ctx = cpdp.cpdp_create(W=2, N=8, tensor_offsets=None, lr=0.1, momentum=0.9, weight_decay=0.0, K=K,
                           slowmo_beta=0.5)
    try:
        cpdp.cpdp_set_method(ctx, cpdp.METHODS[method])
        got = cpdp.lib().cpdp_is_sync_step(ctx, t, T)
        if not 1 <= t <= T:
            assert got == -1
        else:
            assert got == int(method == "ddp" or t % K == 0 or t == T)
    finally:
        cpdp.cpdp_destroy(ctx)


@settings(max_examples=150, deadline=None)
@given(steps=st.integers(1, 50), epochs=st.integers(1, 30), data=st.data(),
       base=st.floats(1e-6, 10.0), frac=st.floats(0.0, 1.0))
def test_schedule_matches_the_oracle(oracle_lib, steps, epochs, data, base, frac):
    warm = data.draw(st.integers(0, epochs - 1))
    K = data.draw(st.integers(1, 8))
    lo = f32(f32(base) * frac)
    ctx = cpdp.cpdp_create(W=2, N=8, tensor_offsets=None, lr=0.1, momentum=0.9, weight_decay=0.0, K=K,
                           slowmo_beta=0.5)
    try:
        cpdp.cpdp_set_schedule(ctx, steps, epochs, warm, base, lo)
        for _ in range(6):
            e = data.draw(st.integers(0, epochs - 1))
            t = data.draw(st.integers(1, steps))
            s = e * steps + t - 1
            want = f32(oracle_lib.scheduled_lr(f32(base), lo, warm * steps, epochs * steps, s))
            assert cpdp.lib().cpdp_scheduled_lr(ctx, e, t) == want
            assert cpdp.lib().cpdp_is_sync_step_at(ctx, e, t) == oracle_lib.is_sync_step_at(e, t, K, steps, warm)
    finally:
        cpdp.cpdp_destroy(ctx)
