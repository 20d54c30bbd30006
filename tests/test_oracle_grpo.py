"""Pins for the masked GRPO loss oracle (Eq. 17 without KL): hand-computed
cases, the on-policy and no-clipping closed forms, masking and normaliser
semantics, central finite differences and torch fp64 autograd."""

import math

import numpy as np
import pytest

from oracle.grpo import grpo_masked_loss


def test_hand_computed_two_tokens():
    # rho = 1.5 and 0.5, eps = 0.2, one response with A = +1, both tokens counted.
    lp = np.log([1.5, 0.5])
    lb = np.zeros(2)
    out = grpo_masked_loss(lp, lb, None, np.array([0, 2]), np.array([1.0]), np.array([1]), 0.2, 0.2)
    # min(1.5, 1.2) = 1.2 (clipped), min(0.5, 0.8) = 0.5 (unclipped): L = -(1.2 + 0.5) / 2
    assert out["loss"] == pytest.approx(-0.85, abs=1e-15)
    np.testing.assert_allclose(out["grad_logp"], [0.0, -0.25], atol=1e-15)
    np.testing.assert_array_equal(out["clipped"], [True, False])
    # A = -1: min(-1.5, -1.2) = -1.5 (unclipped), min(-0.5, -0.8) = -0.8 (clipped)
    neg = grpo_masked_loss(lp, lb, None, np.array([0, 2]), np.array([-1.0]), np.array([1]), 0.2, 0.2)
    assert neg["loss"] == pytest.approx(1.15, abs=1e-15)
    np.testing.assert_allclose(neg["grad_logp"], [0.75, 0.0], atol=1e-15)


def test_asymmetric_clip_range():
    lp = np.log([1.25, 0.85])
    out = grpo_masked_loss(lp, np.zeros(2), None, np.array([0, 2]), np.array([1.0]), np.array([1]),
                           eps_low=0.1, eps_high=0.28)
    # 1.25 < 1 + 0.28: unclipped; 0.85 < 1 - 0.1 = 0.9: min(0.85, 0.9) = 0.85 unclipped.
    assert out["loss"] == pytest.approx(-(1.25 + 0.85) / 2, abs=1e-15)
    assert not out["clipped"].any()


def test_on_policy_closed_form():
    rng = np.random.default_rng(0)
    lens = [5, 9, 3, 7]
    cu = np.concatenate([[0], np.cumsum(lens)])
    lp = rng.normal(-2, 1, cu[-1])
    A = rng.normal(0, 1, 4)
    keep = np.array([1, 0, 1, 1])
    out = grpo_masked_loss(lp, lp, None, cu, A, keep, 0.2, 0.28)
    Z = sum(k * L for k, L in zip(keep, lens))
    assert out["Z"] == Z
    assert out["loss"] == pytest.approx(-sum(k * L * a for k, L, a in zip(keep, lens, A)) / Z, abs=1e-14)
    expect = np.repeat(-keep * A / Z, lens)
    np.testing.assert_allclose(out["grad_logp"], expect, atol=1e-15)


def test_no_clipping_is_plain_importance_weighted_mean():
    rng = np.random.default_rng(1)
    lens = [6, 4]
    cu = np.array([0, 6, 10])
    lp = rng.normal(-2, 1, 10)
    lb = lp + rng.normal(0, 0.5, 10)
    A = np.array([0.7, -1.3])
    out = grpo_masked_loss(lp, lb, None, cu, A, np.array([1, 1]), 1.0 - 1e-12, 1e12)
    rho = np.exp(lp - lb)
    a_tok = np.repeat(A, lens)
    assert out["loss"] == pytest.approx(-(rho * a_tok).sum() / 10, rel=1e-13)
    np.testing.assert_allclose(out["grad_logp"], -rho * a_tok / 10, rtol=1e-13)


def test_masks_normaliser_and_all_dropped():
    lp = np.array([-1.0, -2.0, -3.0, -4.0])
    lb = lp + np.array([0.1, -0.1, 5.0, 0.05])
    mask = np.array([1, 1, 0, 1], dtype=np.uint8)  # token 2 masked: its huge ratio must not count
    cu = np.array([0, 3, 4])
    A = np.array([1.0, -2.0])
    a = grpo_masked_loss(lp, lb, mask, cu, A, np.array([1, 1]), 0.2, 0.2)
    assert a["Z"] == 3 and a["grad_logp"][2] == 0.0
    lp2 = lp.copy()
    lp2[2] = 7.0
    b = grpo_masked_loss(lp2, lb, mask, cu, A, np.array([1, 1]), 0.2, 0.2)
    assert a["loss"] == b["loss"]
    c = grpo_masked_loss(lp, lb, mask, cu, A, np.array([0, 1]), 0.2, 0.2)
    assert c["Z"] == 1 and not c["grad_logp"][:3].any()
    d = grpo_masked_loss(lp, lb, mask, cu, A, np.array([0, 0]), 0.2, 0.2)
    assert d["loss"] == 0.0 and not d["grad_logp"].any()
    assert sum(c["seq_loss"]) == pytest.approx(c["loss"], abs=1e-15)


def test_kl_term_hand_computed_and_identity():
    # one token, rho = 1 (so the surrogate is A = 0.5), reference prob twice the policy's:
    # r = log 2, k = 2 - log 2 - 1; L = -0.5 + beta * k; dL/dlogp = -0.5 + beta * (1 - 2)
    lp = np.array([-1.0])
    lr = lp + np.log(2.0)
    out = grpo_masked_loss(lp, lp, None, np.array([0, 1]), np.array([0.5]), np.array([1]), 0.2, 0.2,
                           logp_ref=lr, beta=0.1)
    k = 1.0 - np.log(2.0)
    assert out["kl"] == pytest.approx(k, abs=1e-15)
    assert out["loss"] == pytest.approx(-0.5 + 0.1 * k, abs=1e-15)
    assert out["grad_logp"][0] == pytest.approx(-0.5 - 0.1, abs=1e-15)
    # reference = policy: the KL term vanishes and changes nothing
    lp2, lb2, mask, cu, A, keep = _random_case(4)
    base = grpo_masked_loss(lp2, lb2, mask, cu, A, keep, 0.2, 0.28)
    same = grpo_masked_loss(lp2, lb2, mask, cu, A, keep, 0.2, 0.28, logp_ref=lp2, beta=0.3)
    assert same["kl"] == 0.0 and same["loss"] == pytest.approx(base["loss"], abs=1e-15)
    np.testing.assert_allclose(same["grad_logp"], base["grad_logp"], atol=1e-15)


def test_kl_estimate_is_nonnegative_and_masked():
    rng = np.random.default_rng(5)
    lp2, lb2, mask, cu, A, keep = _random_case(5)
    lr = lp2 + rng.normal(0, 0.7, lp2.shape[0])
    out = grpo_masked_loss(lp2, lb2, mask, cu, A, keep, 0.2, 0.28, logp_ref=lr, beta=0.05)
    assert out["kl"] > 0.0
    lr2 = lr.copy()
    lr2[~mask.astype(bool)] += 5.0  # masked tokens never count
    assert grpo_masked_loss(lp2, lb2, mask, cu, A, keep, 0.2, 0.28, logp_ref=lr2, beta=0.05)["kl"] == out["kl"]


def _random_case(seed):
    rng = np.random.default_rng(seed)
    lens = [7, 1, 12, 5]
    cu = np.concatenate([[0], np.cumsum(lens)])
    n = cu[-1]
    lp = rng.normal(-2, 1, n)
    lb = lp + rng.normal(0, 0.3, n)
    # keep every ratio at least 1e-3 away from the clip boundaries (the loss is
    # not differentiable there)
    rho = np.exp(lp - lb)
    for bound in (0.8, 1.28):
        near = np.abs(rho - bound) < 1e-3
        lb[near] -= 0.01
    mask = (rng.random(n) < 0.8).astype(np.uint8)
    A = rng.normal(0, 1, len(lens))
    keep = np.array([1, 1, 0, 1])
    return lp, lb, mask, cu, A, keep


@pytest.mark.parametrize("with_kl", [False, True])
def test_gradient_central_differences(with_kl):
    lp, lb, mask, cu, A, keep = _random_case(2)
    lr = lp + np.random.default_rng(9).normal(0, 0.5, lp.shape[0]) if with_kl else None
    beta = 0.2 if with_kl else 0.0

    def loss(x):
        return grpo_masked_loss(x, lb, mask, cu, A, keep, 0.2, 0.28, logp_ref=lr, beta=beta)["loss"]

    out = grpo_masked_loss(lp, lb, mask, cu, A, keep, 0.2, 0.28, logp_ref=lr, beta=beta)
    eps = 1e-7
    fd = np.zeros_like(lp)
    for t in range(lp.shape[0]):
        p, q = lp.copy(), lp.copy()
        p[t] += eps
        q[t] -= eps
        fd[t] = (loss(p) - loss(q)) / (2 * eps)
    np.testing.assert_allclose(out["grad_logp"], fd, atol=1e-8)
    assert out["clipped"].any() and (~out["clipped"] & mask.astype(bool)).any()


def test_gradient_matches_torch_autograd():
    torch = pytest.importorskip("torch")
    lp, lb, mask, cu, A, keep = _random_case(3)
    lr = lp + np.random.default_rng(8).normal(0, 0.4, lp.shape[0])
    out = grpo_masked_loss(lp, lb, mask, cu, A, keep, 0.2, 0.28, logp_ref=lr, beta=0.15)
    t_lp = torch.tensor(lp, requires_grad=True)
    seq = np.repeat(np.arange(len(A)), np.diff(cu))
    a_tok = torch.tensor(A[seq])
    w = torch.tensor(keep[seq] * mask, dtype=torch.float64)
    rho = torch.exp(t_lp - torch.tensor(lb))
    surr = torch.minimum(rho * a_tok, torch.clamp(rho, 0.8, 1.28) * a_tok)
    r = torch.tensor(lr) - t_lp
    kl = torch.exp(r) - r - 1.0
    loss = -(surr * w).sum() / w.sum() + 0.15 * (kl * w).sum() / w.sum()
    loss.backward()
    assert out["loss"] == pytest.approx(loss.item(), abs=1e-14)
    np.testing.assert_allclose(out["grad_logp"], t_lp.grad.numpy(), atol=1e-14)
    assert math.isfinite(out["loss"])
