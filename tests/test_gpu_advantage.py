"""GPU PrimeEcho reward / group advantage (mc_prime_echo_advantages) vs the
fp64 oracle: the paper's batch shape (64 prompts x G = 8, up to K = 3 turns),
the alpha = 1 / alpha = 0 cases, single-turn GRPO (Eq. 3), degenerate
groups, group sizes reduced across warp lanes (dividing 32, with a partial
last warp) and others (one thread per group). Tolerance: 1e-5 absolute on rewards, 1e-4 absolute on advantages
(fp32 two-pass mean / std of O(1) values)."""

import numpy as np
import pytest
import torch

import oracle
from gpu_util import np_
from paper_2606_04847_gb300 import mc

pytestmark = pytest.mark.gpu


def make(T, K, seed):
    g = torch.Generator().manual_seed(seed)
    scores = torch.rand((T, K), generator=g) * 3 - 1
    success = (torch.rand((T, K), generator=g) < 0.35).to(torch.uint8)
    n_turns = torch.randint(1, K + 1, (T,), generator=g, dtype=torch.int32)
    return scores, success, n_turns


def check(scores, success, n_turns, G, alpha, b1, b2, eps):
    out = mc.prime_echo_advantages(scores.cuda(), success.cuda(), n_turns.cuda(), G, alpha, b1, b2, eps)
    torch.cuda.synchronize()
    R = oracle.prime_echo_reward(scores.double().numpy(), success.numpy(), n_turns.numpy(), np.float32(alpha),
                                 np.float32(b1), np.float32(b2))
    A = oracle.group_advantage(R, G, float(np.float32(eps)))
    np.testing.assert_allclose(np_(out["reward"]), R, atol=1e-5)
    np.testing.assert_allclose(np_(out["advantage"]), A, atol=1e-4)
    return out


@pytest.mark.parametrize("alpha", [0.75, 1.0, 0.0])
def test_paper_batch_shape(alpha):
    check(*make(512, 3, 0), 8, alpha, 0.5, 0.2, 1e-6)


def test_single_turn_grpo_advantage():
    scores, success, _ = make(64, 1, 1)
    out = check(scores, success, torch.ones(64, dtype=torch.int32), 8, 0.3, 0.0, 0.0, 1e-6)
    np.testing.assert_allclose(np_(out["reward"]), scores[:, 0].numpy(), atol=1e-6)


def test_degenerate_groups():
    scores = torch.full((16, 2), 0.5)
    success = torch.zeros((16, 2), dtype=torch.uint8)
    out = check(scores, success, torch.full((16,), 2, dtype=torch.int32), 8, 0.75, 0.5, 0.2, 1e-6)
    assert not out["advantage"].any()
    check(*make(5, 3, 2), 1, 0.75, 0.5, 0.2, 1e-6)  # groups of one: advantage 0


@pytest.mark.parametrize("T,G", [(40, 8), (96, 32), (48, 16), (34, 2), (60, 6), (36, 12), (1 << 16, 8),
                                 (24_008, 8), (24_000, 32), (24_001, 1)])  # many 512-row blocks, a partial last
@pytest.mark.parametrize("K", [4, 3])  # 4 turns: vector row loads; 3: per-turn loads
def test_group_sizes_and_batch_tails(T, G, K):
    check(*make(T, K, 3), G, 0.75, 0.5, 0.2, 1e-6)


def test_four_turns_unaligned_rows_take_the_scalar_path():
    scores, success, n_turns = make(65, 4, 4)
    sc = torch.empty(65 * 4 + 1).cuda()[1:].view(65, 4)  # rows 4 bytes off a 16-byte boundary
    sc.copy_(scores.cuda())
    out = mc.prime_echo_advantages(sc, success.cuda(), n_turns.cuda(), 5, 0.75, 0.5, 0.2, 1e-6)
    ref = mc.prime_echo_advantages(scores.cuda(), success.cuda(), n_turns.cuda(), 5, 0.75, 0.5, 0.2, 1e-6)
    torch.cuda.synchronize()
    torch.testing.assert_close(out["advantage"], ref["advantage"], rtol=0, atol=1e-6)
