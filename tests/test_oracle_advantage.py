"""Pins for the PrimeEcho reward / group advantage oracle: the paper's own
special cases (alpha = 1 and alpha = 0, Eq. 11), the early-success bonus
cases, hand-computed values, and the normalisation invariants."""

import numpy as np
import pytest

from oracle.advantage import group_advantage, prime_echo_reward


def test_alpha_one_and_zero_special_cases():
    """Eq. 11: alpha = 1 gives the first-turn reward, alpha = 0 the best-turn
    reward, each plus the early bonus."""
    rng = np.random.default_rng(0)
    T, K = 12, 3
    s = rng.uniform(-1, 2, (T, K))
    ok = rng.random((T, K)) < 0.4
    nt = rng.integers(1, K + 1, T)
    b = prime_echo_reward(s, ok, nt, 1.0, 0.3, 0.1) - prime_echo_reward(s, ok, nt, 1.0, 0.0, 0.0)
    np.testing.assert_allclose(prime_echo_reward(s, ok, nt, 1.0, 0.0, 0.0), s[:, 0], atol=1e-15)
    best = np.array([s[i, :nt[i]].max() for i in range(T)])
    np.testing.assert_allclose(prime_echo_reward(s, ok, nt, 0.0, 0.3, 0.1), best + b, atol=1e-15)


def test_early_success_bonus_cases():
    s = np.zeros((4, 3))
    ok = np.array([[1, 0, 0], [0, 1, 0], [0, 0, 1], [1, 1, 1]], dtype=bool)
    nt = np.array([1, 2, 3, 3])
    R = prime_echo_reward(s, ok, nt, 0.75, 0.5, 0.2)
    # first-turn success: beta1; second-turn success only: beta2; later: none
    np.testing.assert_allclose(R, [0.5, 0.2, 0.0, 0.5], atol=1e-15)
    # a second turn that never ran did not succeed
    R1 = prime_echo_reward(np.zeros((1, 3)), np.array([[0, 1, 1]], bool), np.array([1]), 0.75, 0.5, 0.2)
    assert R1[0] == 0.0


def test_earlier_success_never_earns_less():
    """Eq. 10 with beta1 > beta2 >= 0 (the paper's condition): among
    trajectories with the same per-turn scores that succeed, succeeding at
    turn 1 earns at least as much as first succeeding at turn 2, which earns
    at least as much as first succeeding later."""
    rng = np.random.default_rng(7)
    for _ in range(200):
        K = int(rng.integers(3, 6))
        scores = rng.uniform(-1.0, 2.0, size=(1, K)).repeat(3, axis=0)
        ok = np.zeros((3, K), dtype=bool)
        ok[0, 0] = True                      # first success at turn 1
        ok[1, 1] = True                      # first success at turn 2
        ok[2, int(rng.integers(2, K))] = True  # first success later
        b2 = float(rng.uniform(0.0, 1.0))
        b1 = b2 + float(rng.uniform(1e-3, 1.0))
        R = prime_echo_reward(scores, ok, np.full(3, K), float(rng.uniform(0, 1)), b1, b2)
        assert R[0] > R[1] >= R[2]


def test_hand_computed_reward():
    # alpha = 0.75, scores (-0.5, 0.25, 1.0) over 3 turns, success at turn 3 only:
    # 0.75 * -0.5 + 0.25 * 1.0 + 0 = -0.125
    R = prime_echo_reward(np.array([[-0.5, 0.25, 1.0]]), np.array([[0, 0, 1]], bool), np.array([3]),
                          0.75, 0.5, 0.2)
    assert R[0] == pytest.approx(-0.125, abs=1e-15)


def test_group_advantage_invariants():
    rng = np.random.default_rng(1)
    r = rng.normal(0, 2, 48)
    A = group_advantage(r, 8, 1e-6)
    for g in range(6):
        grp = A[8 * g:8 * g + 8]
        assert abs(grp.mean()) < 1e-12
        assert grp.std(ddof=1) == pytest.approx(1.0, rel=1e-5)
    # shift / positive-scale invariance within a group (eps aside)
    np.testing.assert_allclose(group_advantage(3 * r + 5, 8, 0.0), group_advantage(r, 8, 0.0), atol=1e-12)


def test_group_advantage_hand_computed_and_degenerate():
    A = group_advantage(np.array([1.0, 2.0, 3.0, 6.0]), 4, 0.0)
    # mean 3, sample std sqrt((4 + 1 + 0 + 9) / 3)
    sd = np.sqrt(14.0 / 3.0)
    np.testing.assert_allclose(A, np.array([-2.0, -1.0, 0.0, 3.0]) / sd, atol=1e-15)
    np.testing.assert_allclose(group_advantage(np.full(8, 0.7), 8, 1e-6), 0.0, atol=1e-12)
    np.testing.assert_allclose(group_advantage(np.array([5.0, -1.0]), 1, 1e-6), 0.0, atol=1e-15)
    with pytest.raises(ValueError):
        group_advantage(np.zeros(5), 4, 1e-6)
