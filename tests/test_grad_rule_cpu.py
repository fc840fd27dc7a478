"""CPU: the coefficient-gradient comparison rule of the GPU parity tests
(gpu_helpers.assert_grad_close) accepts what the rule allows and rejects
planted departures from it: a gradient off by more than 1e-5 relative, a
non-finite value where no binary32 intermediate can overflow, a finite value
where the exact gradient is beyond the binary32 range, and a finite but
wrong value in the range where an overflow is allowed."""
import numpy as np
import pytest

from gpu_helpers import FLOOR_ROW, OVERFLOW_ABS, assert_grad_close


def _case():
    ref = np.array([1.0, -2.0, 3.0e-3, 0.0], np.float32)
    ref_abs = np.array([1.5, 2.0, 4.0, 1.0e-3])
    return ref, ref_abs


def test_accepts_within_tolerance():
    ref, ref_abs = _case()
    got = ref.astype(np.float64) * (1 + 0.9e-5)
    assert_grad_close(got.astype(np.float32), ref, ref_abs, FLOOR_ROW, "ok")


def test_rejects_relative_error():
    ref, ref_abs = _case()
    got = ref.copy()
    got[1] = np.float32(-2.0 * (1 + 3e-5))
    with pytest.raises(AssertionError, match="outside tolerance"):
        assert_grad_close(got, ref, ref_abs, FLOOR_ROW, "planted")


def test_rejects_nan_where_nothing_overflows():
    ref, ref_abs = _case()
    got = ref.copy()
    got[2] = np.nan
    with pytest.raises(AssertionError, match="nothing can overflow"):
        assert_grad_close(got, ref, ref_abs, FLOOR_ROW, "planted")


def test_rejects_finite_beyond_range():
    ref, ref_abs = _case()
    ref[0] = np.inf
    ref_abs[0] = 4.0e38
    got = ref.copy()
    got[0] = np.float32(3.0e38)
    with pytest.raises(AssertionError, match="beyond the binary32 range"):
        assert_grad_close(got, ref, ref_abs, FLOOR_ROW, "planted")
    got[0] = np.inf
    assert_grad_close(got, ref, ref_abs, FLOOR_ROW, "non-finite is right")


def test_overflow_range_allows_nan_but_checks_finite_values():
    ref = np.array([0.0, 5.0], np.float32)
    ref_abs = np.array([2.0 ** 129, 2.0 ** 127])
    assert ref_abs.min() > OVERFLOW_ABS
    assert_grad_close(np.array([np.nan, np.nan], np.float32), ref, ref_abs, FLOOR_ROW, "nan allowed")
    assert_grad_close(np.array([0.0, 5.0], np.float32), ref, ref_abs, FLOOR_ROW, "exact")
    # finite there, it must still be within the bound (floor * 2^129 = 2^89)
    with pytest.raises(AssertionError, match="outside tolerance"):
        assert_grad_close(np.array([2.0 ** 100, 5.0], np.float32), ref, ref_abs, FLOOR_ROW, "planted")
