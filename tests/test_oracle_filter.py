"""Pins for the fp64 oracle of the sequence ratio statistics and MirrorPop mask.

Checked against the paper's worked example (tests/golden), the product forms
of Eq. 18 and Eq. 20 evaluated with Python's math module, closed forms
(constant gap, identical policies), the triangle inequality, masking
semantics and the "<=" threshold of Eq. 21.
"""

import json
import math
import os

import numpy as np
import pytest

from oracle.filter import seq_ratio_filter

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "mirrorpop_worked_example.json")


def test_paper_worked_example():
    ex = json.load(open(GOLDEN))
    rho = np.array(ex["rho"])
    lp_pi = np.log(rho) - 3.0          # any policy log-probs with the stated ratios
    lp_b = np.full(2, -3.0)
    out = seq_ratio_filter(lp_pi, lp_b, None, np.array([0, 2]), delta=0.5, delta_vanilla=0.5)
    assert abs(out["signed_mean"][0] - ex["signed_mean_log_ratio"]) < 1e-15
    assert abs(math.exp(out["signed_mean"][0]) - ex["geometric_mean_ratio"]) < 1e-15
    assert abs(out["abs_mean"][0] - ex["abs_mean_log_ratio"]) < 1e-15
    assert abs(math.exp(out["abs_mean"][0]) - ex["mirror_ratio_magnitude"]) < 1e-13
    mirror = np.maximum(out["token_ratio"], 1.0 / out["token_ratio"])
    np.testing.assert_allclose(mirror, ex["mirror_deviation_per_token"], rtol=1e-14)
    # The Vanilla statistic calls this sequence on-policy, MirrorPop drops it.
    assert out["keep_vanilla"][0] == 1 and out["keep"][0] == 0


def test_product_forms_of_eq18_and_eq20():
    """exp(S) = (prod rho)^(1/L) and exp(A) = (prod max(rho, 1/rho))^(1/L),
    evaluated directly with Python floats on short sequences."""
    rng = np.random.default_rng(0)
    lens = [1, 3, 7, 12]
    cu = np.concatenate([[0], np.cumsum(lens)])
    lp_pi = rng.normal(-2.0, 1.0, cu[-1])
    lp_b = lp_pi + rng.normal(0, 0.4, cu[-1])
    out = seq_ratio_filter(lp_pi, lp_b, None, cu, delta=0.3)
    for i, L in enumerate(lens):
        rho = [math.exp(a) / math.exp(b) for a, b in zip(lp_pi[cu[i]:cu[i + 1]], lp_b[cu[i]:cu[i + 1]])]
        geo = math.prod(rho) ** (1.0 / L)
        mir = math.prod(max(r, 1.0 / r) for r in rho) ** (1.0 / L)
        assert abs(math.exp(out["signed_mean"][i]) / geo - 1) < 1e-13
        assert abs(math.exp(out["abs_mean"][i]) / mir - 1) < 1e-13
        assert out["keep"][i] == (1 if math.log(mir) <= 0.3 else 0)
        np.testing.assert_allclose(out["token_ratio"][cu[i]:cu[i + 1]], rho, rtol=1e-14)


def test_identical_policies_keep_everything():
    rng = np.random.default_rng(1)
    lp = rng.normal(-3, 2, 40)
    out = seq_ratio_filter(lp, lp.copy(), None, np.array([0, 10, 25, 40]), delta=0.0,
                           delta_vanilla=0.0)
    assert not np.any(out["signed_mean"]) and not np.any(out["abs_mean"])
    assert np.all(out["keep"] == 1) and np.all(out["keep_vanilla"] == 1)
    np.testing.assert_array_equal(out["token_ratio"], 1.0)
    np.testing.assert_array_equal(out["token_keep"], 1)


def test_constant_gap_and_triangle_inequality():
    rng = np.random.default_rng(2)
    lens = rng.integers(1, 50, 20)
    cu = np.concatenate([[0], np.cumsum(lens)])
    lp_pi = rng.normal(-2, 1, cu[-1])
    gaps = rng.normal(0, 0.3, 20)
    lp_b = lp_pi - np.repeat(gaps, lens)
    out = seq_ratio_filter(lp_pi, lp_b, None, cu, delta=0.2)
    np.testing.assert_allclose(out["signed_mean"], gaps, atol=1e-14)
    np.testing.assert_allclose(out["abs_mean"], np.abs(gaps), atol=1e-14)
    np.testing.assert_array_equal(out["n_tokens"], lens)
    noisy = seq_ratio_filter(lp_pi, lp_pi + rng.normal(0, 0.5, cu[-1]), None, cu, 0.2, 0.2)
    assert np.all(np.abs(noisy["signed_mean"]) <= noisy["abs_mean"] + 1e-15)
    # MirrorPop keep implies Vanilla keep at equal thresholds.
    assert np.all(noisy["keep"] <= noisy["keep_vanilla"])


def test_loss_mask_semantics_and_empty_sequences():
    lp_pi = np.array([0.0, -1.0, -2.0, -3.0, -4.0, -5.0])
    lp_b = np.array([0.5, -1.5, 9.0, -3.0, -4.0, -5.0])
    mask = np.array([1, 1, 0, 0, 0, 1], dtype=np.uint8)
    # seq 0 = tokens 0..2 (token 2 masked: its huge gap must not count)
    # seq 1 = tokens 3..4 (all masked: L = 0), seq 2 = token 5, seq 3 = empty
    cu = np.array([0, 3, 5, 6, 6])
    out = seq_ratio_filter(lp_pi, lp_b, mask, cu, delta=0.5, delta_vanilla=0.1)
    np.testing.assert_array_equal(out["n_tokens"], [2, 0, 1, 0])
    np.testing.assert_allclose(out["signed_mean"], [0.0, 0, 0, 0], atol=1e-15)
    np.testing.assert_allclose(out["abs_mean"], [0.5, 0, 0, 0], atol=1e-15)
    # "<=" keeps A = delta exactly (0.5 is exact in binary).
    np.testing.assert_array_equal(out["keep"], [1, 0, 1, 0])
    np.testing.assert_array_equal(out["keep_vanilla"], [1, 0, 1, 0])
    np.testing.assert_array_equal(out["token_keep"], [1, 1, 0, 0, 0, 1])


def test_vanilla_not_requested():
    lp = np.zeros(4)
    out = seq_ratio_filter(lp, lp, None, np.array([0, 4]), delta=0.1, delta_vanilla=-1.0)
    assert out["keep"][0] == 1 and out["keep_vanilla"][0] == 0


def test_bad_cu_seqlens():
    with pytest.raises(ValueError):
        seq_ratio_filter(np.zeros(3), np.zeros(3), None, np.array([0, 2]), 0.1)
    with pytest.raises(ValueError):
        seq_ratio_filter(np.zeros(3), np.zeros(3), None, np.array([0, 2, 1, 3]), 0.1)
