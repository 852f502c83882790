"""The weight bar of the GPU parity tests (tests/parity.py), checked on the
CPU: it accepts the fp32 rounding a correct kernel makes and rejects the
errors a wrong one would.

The floor of the relative error is max(|W|, lr, |W_t - W_{t-1}|): lr stands
for the size of one update lr |u| when |u| ~ 1; without bias correction
(the ablation of Section 2.1) |u| reaches 1/sqrt(1 - beta2^t), and the
oracle's own step is the size to compare with.
"""
import numpy as np
import pytest

from parity import check_weights


def test_fp32_near_cancellation_within_fp32_error_of_the_step_passes():
    lr = 2e-3
    prev = np.array([0.0629, 0.01], np.float32)
    step = np.array([-0.0629 + 1.8e-6, 1e-3], np.float64)  # |u| ~ 31 on the first element
    want = (prev.astype(np.float64) + step).astype(np.float32)
    got = want.copy()
    got[0] += np.float32(2.2e-8)  # about 6 fp32 ulps of the step
    with pytest.raises(AssertionError):
        check_weights(got, want, lr)  # floor lr: 1.1e-5 of lr
    check_weights(got, want, lr, prev=prev)


def test_fp32_error_of_1e4_of_the_step_fails():
    lr = 2e-3
    prev = np.array([0.0629], np.float32)
    want = np.array([1.8e-6], np.float32)
    got = want + np.float32(1e-4 * 0.0629)
    with pytest.raises(AssertionError):
        check_weights(got, want, lr, prev=prev)


def test_fp32_wrong_update_on_ordinary_elements_fails():
    rng = np.random.default_rng(0)
    lr = 1e-3
    prev = (rng.standard_normal(1000) * 0.02).astype(np.float32)
    want = (prev - lr * np.sign(rng.standard_normal(1000))).astype(np.float32)
    got = want.copy()
    got[17] = prev[17] - 1.001 * (prev[17] - want[17])  # a step 0.1 % too long
    with pytest.raises(AssertionError):
        check_weights(got, want, lr, prev=prev)


def test_bf16_near_cancellation_uses_the_step_floor():
    """bf16 W: an element 3 ulps off where the new weight nearly cancels is
    within fp32 error of a 0.06 step, not of lr; a 0.1 % longer step on an
    ordinary element is more than 1 ulp and fails."""
    import oracle
    lr = 2e-3
    prev = oracle.round_bf16(np.array([0.0629, 0.02]))
    want = oracle.round_bf16(np.array([-1.7956e-6, 0.021]))
    got = want.copy()
    got[0] += 3  # same sign, 3 ulps further from zero
    with pytest.raises(AssertionError):
        check_weights(got, want, lr)
    check_weights(got, want, lr, prev=prev)
    far = want.copy()
    far[1] += 2
    with pytest.raises(AssertionError):
        check_weights(far, want, lr, prev=prev)


def test_bf16_beyond_one_ulp_only_where_the_step_cancels_the_weight():
    """Two ulps off on a small weight that the step does not cancel fails,
    however few such elements there are: the near-cancellation set
    (|W_t| <= 2^-12 of the step) is the only place a correct fp32 update can
    land more than one bf16 ulp from the oracle."""
    import oracle
    lr = 1e-3
    prev = oracle.round_bf16(np.full(100000, 0.02))
    want = oracle.round_bf16(np.concatenate([[2e-5], np.full(99999, 0.019)]))
    got = want.copy()
    got[0] += 2  # |W_t| = 2e-5 against a 0.02 step: 1e-3 of it, not cancelling
    with pytest.raises(AssertionError):
        check_weights(got, want, lr, prev=prev)
    want[0] = oracle.round_bf16(np.array([6e-6]))[0]  # 3e-4 of the step: still outside 2^-12
    got[0] = want[0] + 2
    with pytest.raises(AssertionError):
        check_weights(got, want, lr, prev=prev)
    want[0] = oracle.round_bf16(np.array([4e-7]))[0]  # 2e-5 of the step: inside 2^-12
    got[0] = want[0] + 2
    check_weights(got, want, lr, prev=prev)
