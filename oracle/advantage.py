"""Oracle: PrimeEcho trajectory reward and the group-normalised advantage.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): never imported by the
product path. NumPy float64, one trajectory / one group at a time.

Paper passages followed (§4.4.3, §4.4.1)
---------------------------------------
* Eq. 9: R_i = alpha s_{i,1} + (1 - alpha) max_{1<=k<=K_i} s_{i,k} + b_early(i),
  s_{i,k} the score of turn k of trajectory i.
* Eq. 10: b_early(i) = beta1 1[success_{i,1}] + beta2 1[not success_{i,1} and
  success_{i,2}].
* Eq. 12 (and Eq. 3 for single-turn rewards): A_i = (R_i - mean_G R) /
  (std_G R + eps) over the G trajectories of the same prompt.

Readings where the paper is silent
----------------------------------
* A trajectory that stopped after K_i < K turns has turns K_i+1..K absent:
  the max runs over its K_i turns and a second turn that never ran did not
  succeed. K_i >= 1.
* std is the sample standard deviation (divisor G - 1), as GRPO
  implementations compute it; a group of one has std 0 (and A = 0).
* Groups are G consecutive trajectories.
"""

from __future__ import annotations

import numpy as np

__all__ = ["prime_echo_reward", "group_advantage"]


def prime_echo_reward(scores, success, n_turns, alpha: float, beta1: float, beta2: float):
    """Eq. 9-10 per trajectory. ``scores`` / ``success`` are [T, K] (turn k of
    trajectory i at [i, k]); ``n_turns`` [T] the turns each trajectory ran."""
    s = np.asarray(scores, dtype=np.float64)
    ok = np.asarray(success).astype(bool)
    nt = np.asarray(n_turns, dtype=np.int64)
    T = s.shape[0]
    R = np.zeros(T)
    for i in range(T):
        k = int(nt[i])
        best = max(s[i, j] for j in range(k))
        first_ok = bool(ok[i, 0])
        second_ok = k >= 2 and bool(ok[i, 1])
        b = beta1 * (1.0 if first_ok else 0.0) + beta2 * (1.0 if (not first_ok and second_ok) else 0.0)
        R[i] = alpha * s[i, 0] + (1.0 - alpha) * best + b
    return R


def group_advantage(rewards, group_size: int, eps: float):
    """Eq. 12 / Eq. 3 over consecutive groups of ``group_size`` trajectories."""
    r = np.asarray(rewards, dtype=np.float64)
    if r.shape[0] % group_size:
        raise ValueError("the number of trajectories must be a multiple of the group size")
    A = np.zeros_like(r)
    for g0 in range(0, r.shape[0], group_size):
        grp = r[g0:g0 + group_size]
        mean = grp.sum() / group_size
        std = np.sqrt(((grp - mean) ** 2).sum() / (group_size - 1)) if group_size > 1 else 0.0
        A[g0:g0 + group_size] = (grp - mean) / (std + eps)
    return A
