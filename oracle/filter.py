"""Oracle: per-sequence importance-ratio statistics and the MirrorPop keep-mask.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): never imported by the
product path. NumPy float64 on the CPU, one sequence at a time.

Paper passages followed (§4.4.1 and §4.5.2)
-------------------------------------------
* Eq. 4: token importance ratio  rho_{i,t} = pi_theta / pi_rollout, here from
  per-token log-probs: log rho_{i,t} = logp_policy_t - logp_behaviour_t.
* Eq. 18: the conventional sequence statistic, the geometric mean of the token
  ratios, equal to exp of the signed mean log-ratio
      S_i = (1/L_i) sum_t log rho_{i,t}.
* Eq. 19: the mirror deviation m_{i,t} = max(rho, 1/rho) = exp(|log rho|).
* Eq. 20: the MirrorPop statistic, exp of the absolute mean log-ratio
      A_i = (1/L_i) sum_t |log rho_{i,t}|.
* Eq. 21: the keep-mask M_i = 1[A_i <= delta], delta in log-ratio space.
* §5.4.6 reports both S_i and A_i as passive diagnostics; they are outputs.

Readings where the paper is silent
----------------------------------
* Which tokens count (L_i): the tokens of sequence i whose loss_mask is 1
  (the caller decides, e.g. response tokens only). No mask = every token.
* L_i = 0: S_i = A_i = 0 and keep_i = 0 (the sequence contributes nothing).
* The conventional ("Vanilla") trust interval is not given numerically; it is
  read as symmetric in log space: keep_vanilla_i = 1[|S_i| <= delta_vanilla].
  A negative delta_vanilla means "not requested".
* The threshold comparison is "<=", as Eq. 21 writes it.
* The per-token outputs are rho_t = exp(log rho_t) and
  token_keep_t = keep_{seq(t)} AND loss_mask_t.
"""

from __future__ import annotations

import numpy as np

from .logprobs import as_f64, as_i64

__all__ = ["seq_ratio_filter"]


def _as_mask(loss_mask, n):
    if loss_mask is None:
        return np.ones(n, dtype=bool)
    if hasattr(loss_mask, "detach"):
        loss_mask = loss_mask.detach().cpu().numpy()
    return np.asarray(loss_mask).astype(bool)


def seq_ratio_filter(logp_policy, logp_behaviour, loss_mask, cu_seqlens,
                     delta: float, delta_vanilla: float = -1.0):
    """Per-sequence S_i, A_i, L_i, MirrorPop keep_i (+ Vanilla keep) and per-token ratios.

    ``cu_seqlens`` is the [B+1] prefix of sequence lengths over the packed
    token arrays. Returns a dict of NumPy arrays:
    ``signed_mean`` [B], ``abs_mean`` [B], ``n_tokens`` [B] (int64),
    ``keep`` [B] (uint8), ``keep_vanilla`` [B] (uint8; all 0 when not requested),
    ``token_ratio`` [N], ``token_keep`` [N] (uint8).
    """
    lp = as_f64(logp_policy)
    lb = as_f64(logp_behaviour)
    cu = as_i64(cu_seqlens)
    n = lp.shape[0]
    mask = _as_mask(loss_mask, n)
    B = cu.shape[0] - 1
    if cu[0] != 0 or cu[-1] != n or np.any(np.diff(cu) < 0):
        raise ValueError("cu_seqlens must start at 0, end at N and be non-decreasing")

    log_rho = lp - lb                      # Eq. 4, in log space
    token_ratio = np.exp(log_rho)          # rho_t itself
    S = np.zeros(B)
    A = np.zeros(B)
    L = np.zeros(B, dtype=np.int64)
    keep = np.zeros(B, dtype=np.uint8)
    keep_v = np.zeros(B, dtype=np.uint8)
    token_keep = np.zeros(n, dtype=np.uint8)
    for i in range(B):
        sl = slice(cu[i], cu[i + 1])
        sel = log_rho[sl][mask[sl]]
        L[i] = sel.shape[0]
        if L[i] == 0:
            continue
        S[i] = sel.sum() / L[i]             # exponent of Eq. 18
        A[i] = np.abs(sel).sum() / L[i]     # exponent of Eq. 20
        keep[i] = 1 if A[i] <= delta else 0                  # Eq. 21
        if delta_vanilla >= 0:
            keep_v[i] = 1 if abs(S[i]) <= delta_vanilla else 0
        token_keep[sl] = keep[i] & mask[sl]
    return {
        "signed_mean": S,
        "abs_mean": A,
        "n_tokens": L,
        "keep": keep,
        "keep_vanilla": keep_v,
        "token_ratio": token_ratio,
        "token_keep": token_keep,
    }
