"""Oracle: the masked GRPO objective and its gradient with respect to the
policy log-probs. NumPy float64, one sequence at a time.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): never imported by the
product path.

Paper passages followed
-----------------------
* Eq. 4 (§4.4.1): rho_{i,t} = pi_theta / pi_rollout, here exp(logp_policy -
  logp_behaviour).
* Eq. 5 (§4.4.1) and Eq. 17 (§4.5.2): the clipped surrogate
      s_{i,t} = min(rho A_i, clip(rho, 1 - eps_low, 1 + eps_high) A_i)
  summed over the tokens of every response, each response multiplied by its
  mask M_i, normalised by sum_i M_i L_i, negated:
      L = -(1 / sum_i M_i L_i) sum_i sum_t s_{i,t} M_i  +  beta KL.
* The beta * KL(pi_theta || pi_ref) term of Eq. 5 / Eq. 17, estimated per
  token from the sampled token's log-probs (the paper does not fix the
  estimator; this is the non-negative per-token estimator used with GRPO):
      k_t = pi_ref / pi_theta - log(pi_ref / pi_theta) - 1 = e^r - r - 1,
      r = logp_ref_t - logp_policy_t,
  averaged with the same mask and normaliser as the surrogate:
      KL = (1 / sum_i M_i L_i) sum_i M_i sum_t k_t.

Readings where the paper is silent
----------------------------------
* L_i and the tokens summed are those with loss_mask = 1 (as in the filter).
* sum_i M_i L_i = 0 (every response dropped): L = 0 and a zero gradient.
* Gradient: d s / d logp = rho A when the minimum is attained by the
  unclipped term rho A (including ties, i.e. whenever rho lies inside the
  clip range), and 0 when the clipped term is strictly smaller.
"""

from __future__ import annotations

import numpy as np

from .logprobs import as_f64, as_i64

__all__ = ["grpo_masked_loss"]


def _mask(x, n):
    if x is None:
        return np.ones(n, dtype=bool)
    if hasattr(x, "detach"):
        x = x.detach().cpu().numpy()
    return np.asarray(x).astype(bool)


def grpo_masked_loss(logp_policy, logp_behaviour, loss_mask, cu_seqlens, advantages, keep,
                     eps_low: float, eps_high: float, logp_ref=None, beta: float = 0.0):
    """Masked GRPO loss (Eq. 17) and dL/dlogp_policy.

    ``advantages`` [B] are the response-level advantages A_i (Eq. 3),
    ``keep`` [B] the masks M_i (Eq. 21); ``logp_ref`` [N] (optional) the
    reference policy's log-probs for the beta * KL term. Returns a dict with
    ``loss`` (float), ``grad_logp`` [N], ``seq_loss`` [B] (each response's
    share of ``loss``), ``kl`` (the masked mean KL estimate, before beta),
    ``clipped`` [N] (bool: the clipped term was strictly smaller) and ``Z``.
    """
    lp = as_f64(logp_policy)
    lb = as_f64(logp_behaviour)
    cu = as_i64(cu_seqlens)
    A = as_f64(advantages)
    M = _mask(keep, A.shape[0]).astype(np.float64)
    n = lp.shape[0]
    m = _mask(loss_mask, n)
    B = cu.shape[0] - 1
    L = np.array([m[cu[i]:cu[i + 1]].sum() for i in range(B)], dtype=np.float64)
    Z = float((M * L).sum())
    lr = None if logp_ref is None else as_f64(logp_ref)
    grad = np.zeros(n)
    seq_loss = np.zeros(B)
    kl_total = 0.0
    clipped = np.zeros(n, dtype=bool)
    if Z == 0.0:
        return {"loss": 0.0, "grad_logp": grad, "seq_loss": seq_loss, "kl": 0.0, "clipped": clipped, "Z": Z}
    for i in range(B):
        for t in range(cu[i], cu[i + 1]):
            if not m[t]:
                continue
            rho = np.exp(lp[t] - lb[t])                                   # Eq. 4
            unclipped = rho * A[i]
            clipped_term = np.clip(rho, 1.0 - eps_low, 1.0 + eps_high) * A[i]
            s = min(unclipped, clipped_term)                              # Eq. 5 / 17
            seq_loss[i] -= s * M[i] / Z
            if clipped_term < unclipped:
                clipped[t] = True
            elif M[i] != 0.0:
                grad[t] = -M[i] * rho * A[i] / Z
            if lr is not None:
                r = lr[t] - lp[t]
                k = np.exp(r) - r - 1.0                                   # KL estimate per token
                kl_total += M[i] * k / Z
                seq_loss[i] += beta * M[i] * k / Z
                grad[t] += beta * M[i] * (1.0 - np.exp(r)) / Z            # d k / d logp_policy
    return {"loss": float(seq_loss.sum()), "grad_logp": grad, "seq_loss": seq_loss, "kl": float(kl_total),
            "clipped": clipped, "Z": Z}
