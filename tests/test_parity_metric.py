"""The parity metric itself (tests/parity.py), on hand-made values: the base
denominator, the capped parameter floor, the history scale, and the
statistics run_and_check reports. No GPU."""
import numpy as np

from parity import TOL, error_stats


def test_base_denominator_is_element_or_tensor_rms():
    ref = np.array([[1.0, 1e-6, -1.0, 0.0]])
    x = ref + np.array([[0.0, 5e-6, 0.0, 0.0]])
    st = error_stats(x, ref, np.array([0, 0, 0, 0]))
    rms = np.sqrt(np.mean(ref * ref))
    assert np.isclose(st.err, 5e-6 / rms) and st.err == st.plain and st.governed == 0


def test_parameter_floor_is_capped():
    ref = np.array([[1e-3]])
    x = ref + 1e-6                        # 1e-3 relative: a real mistake
    raw = error_stats(x, ref, np.array([0]))
    assert raw.err > TOL
    capped = error_stats(x, ref, np.array([0]), floor=np.array([1.0]), cap=10.0)
    assert np.isclose(capped.err, 1e-6 / (10.0 * 1e-3)) and capped.err > TOL
    assert capped.governed == 1 and np.isclose(capped.max_ratio, 1000.0) and capped.plain == raw.plain


def test_history_scale_absorbs_carried_rounding_not_a_mistake():
    """A one-element tensor that started at 3.6e-3 and cancelled to -1.6e-6:
    float32 carried about 3 ulps of its starting magnitude (8e-10), which is a
    5e-4 relative error at its current value. Against the history scale (the
    largest magnitude it had) that is 2.3e-7; an error of a mistake's size
    (1e-7 absolute, 30 ulps of the start) still fails."""
    tid, hist = np.array([0]), np.array([3.5653829e-3])
    ref = np.array([[-1.5929895397693195e-06]])
    carried = np.array([[-1.5921832527965307e-06]])
    assert error_stats(carried, ref, tid).err > TOL
    st = error_stats(carried, ref, tid, hist=hist)
    assert st.err < TOL and st.plain > TOL and st.governed == 1 and st.max_ratio > 1000.0
    wrong = ref + 1e-7
    assert error_stats(wrong, ref, tid, hist=hist).err > TOL


def test_history_scale_changes_nothing_while_the_scale_holds():
    rng = np.random.default_rng(0)
    ref = rng.normal(size=(2, 100))
    x = ref * (1.0 + 1e-7)
    tid = np.repeat(np.arange(4), 25)
    rms = np.array([np.sqrt(np.mean(ref[:, tid == t] ** 2)) for t in range(4)])
    a = error_stats(x, ref, tid)
    b = error_stats(x, ref, tid, hist=rms[tid])
    assert a.err == b.err and b.governed == 0
