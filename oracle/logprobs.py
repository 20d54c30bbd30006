"""Oracle: LM-head projection, log-softmax over the full vocabulary, entropy,
and the closed-form backward. NumPy float64 on the CPU.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): never imported by the
product path.

What the paper fixes
--------------------
The policy probability of the sampled token, pi_theta(o_{i,t} | x, o_{i,<t}),
appears in the token importance ratio (Eq. 4, §4.4.1) and in the GRPO
objective (Eq. 5) and its masked form (Eq. 17, §4.5.2). The paper does not
spell out how it is computed; for a decoder LM it is the softmax over the
vocabulary of the LM-head logits at the sampled token, which is what this module
writes out. Token entropy is tracked as a training diagnostic (the "Entropy"
panel of the MirrorPop ablation, §5.4.6) without a formula; the Shannon entropy
in nats of the same softmax is used.

Definitions (one row t at a time; rows are independent)
--------------------------------------------------------
    z_{t,v}  = (sum_k h_{t,k} w_{v,k}) * inv_temperature
    m_t      = max_v z_{t,v}
    lse_t    = m_t + log sum_v exp(z_{t,v} - m_t)
    logp_t   = z_{t,y_t} - lse_t
    p_{t,v}  = exp(z_{t,v} - lse_t)
    H_t      = -sum_v p_{t,v} log p_{t,v} = lse_t - sum_v p_{t,v} z_{t,v}

This is the two-pass textbook form (max, then sum); it shares nothing with the
kernels' single-pass online update.

Backward. For an upstream scalar  L = sum_t g_t logp_t + sum_t gH_t H_t,
differentiating the definitions above:
    d logp_t / d z_{t,v} = 1[v = y_t] - p_{t,v}
    d H_t    / d z_{t,v} = -p_{t,v} (log p_{t,v} + H_t)
    dZ_{t,v} = inv_temperature * ( g_t (1[v=y_t] - p_{t,v})
                                   - gH_t p_{t,v} (log p_{t,v} + H_t) )
    dL/dh_t  = sum_v dZ_{t,v} w_v           (dH = dZ W)
    dL/dw_v  = sum_t dZ_{t,v} h_t           (dW = dZ^T H)
The inv_temperature factor is the chain rule through z = (h . w) * inv_temperature.

Inputs are bf16 (or any float) arrays; they are upcast exactly to float64.
Rows are processed in independent groups only to bound memory; within a row
nothing is blocked, fused or reordered.
"""

from __future__ import annotations

import numpy as np

__all__ = ["as_f64", "logprob_state", "token_logprobs", "token_logprobs_bwd", "token_logprobs_bwd_rows"]


def as_f64(x) -> np.ndarray:
    """Exact upcast of a torch tensor (any float dtype, incl. bf16) or array to float64."""
    if hasattr(x, "detach"):  # torch.Tensor, without importing torch here
        x = x.detach()
        if x.device.type != "cpu":
            x = x.cpu()
        import torch  # local: the oracle itself is NumPy; torch only converts

        return x.to(torch.float64).numpy()
    return np.asarray(x, dtype=np.float64)


def as_i64(x) -> np.ndarray:
    if hasattr(x, "detach"):
        x = x.detach()
        if x.device.type != "cpu":
            x = x.cpu()
        return x.to(dtype=__import__("torch").int64).numpy()
    return np.asarray(x, dtype=np.int64)


def _row_stats(z: np.ndarray, y: np.ndarray):
    """Two-pass log-softmax statistics of a block of rows of logits z [R, V]."""
    m = z.max(axis=1)
    lse = m + np.log(np.exp(z - m[:, None]).sum(axis=1))
    rows = np.arange(z.shape[0])
    logp = z[rows, y] - lse
    p = np.exp(z - lse[:, None])
    ent = lse - (p * z).sum(axis=1)
    return logp, ent, lse


def token_logprobs(hidden, w_vocab, targets, inv_temperature: float = 1.0,
                   rows_per_block: int = 64, vocab_per_block: int = 32768):
    """Per-row target log-prob, entropy and log-sum-exp (module docstring).

    Returns a dict of float64 arrays ``logp``, ``entropy``, ``lse`` of length N.
    A target outside [0, V) is an error (ValueError): the oracle has no
    "invalid row" convention to check against.
    """
    h = as_f64(hidden)
    y = as_i64(targets)
    n = h.shape[0]
    wsrc = w_vocab
    V = wsrc.shape[0]
    if y.shape != (n,):
        raise ValueError("targets must have shape [N]")
    if n and (y.min() < 0 or y.max() >= V):
        raise ValueError("target out of range [0, V)")
    logp = np.empty(n)
    ent = np.empty(n)
    lse = np.empty(n)
    # W is upcast in vocabulary blocks so a [V, d] float64 copy need not exist.
    wblocks = [(v0, min(V, v0 + vocab_per_block)) for v0 in range(0, V, vocab_per_block)]
    w64 = None
    if len(wblocks) == 1:
        w64 = as_f64(wsrc)
    for r0 in range(0, n, rows_per_block):
        r1 = min(n, r0 + rows_per_block)
        z = np.empty((r1 - r0, V))
        for v0, v1 in wblocks:
            wb = w64 if w64 is not None else as_f64(wsrc[v0:v1])
            z[:, v0:v1] = h[r0:r1] @ wb.T
        z *= float(inv_temperature)
        logp[r0:r1], ent[r0:r1], lse[r0:r1] = _row_stats(z, y[r0:r1])
    return {"logp": logp, "entropy": ent, "lse": lse}


def logprob_state(hidden, w_shard, targets, v_begin: int, inv_temperature: float = 1.0):
    """Softmax state of one vocabulary shard, columns [v_begin, v_begin + V_shard)
    of a larger vocabulary (the rows w_shard of its LM head), per row t:
        m = max_v z_{t,v},  s = sum_v exp(z - m),  t = sum_v exp(z - m)(z - m),
        z_y = z_{t, y_t} if the shard holds y_t, else -inf.
    Returns float64 [N, 4] = (m, s, t, z_y). Over a whole vocabulary,
    lse = m + log s and entropy = log s - t / s (module docstring)."""
    h = as_f64(hidden)
    y = as_i64(targets)
    z = (h @ as_f64(w_shard).T) * float(inv_temperature)
    n, vs = z.shape
    m = z.max(axis=1)
    e = np.exp(z - m[:, None])
    s = e.sum(axis=1)
    t = (e * (z - m[:, None])).sum(axis=1)
    local = y - int(v_begin)
    own = (local >= 0) & (local < vs)
    zy = np.full(n, -np.inf)
    zy[own] = z[np.arange(n)[own], local[own]]
    return np.stack([m, s, t, zy], axis=1)


def token_logprobs_bwd(hidden, w_vocab, targets, grad_logp, grad_entropy=None,
                       inv_temperature: float = 1.0, return_dz: bool = False):
    """Closed-form gradients of L = sum_t g_t logp_t + sum_t gH_t H_t.

    Returns a dict with float64 ``grad_hidden`` [N, d] and ``grad_w`` [V, d]
    (and ``dz`` [N, V] with ``return_dz``). Small problems only: Z is formed
    whole.
    """
    h = as_f64(hidden)
    w = as_f64(w_vocab)
    y = as_i64(targets)
    g = as_f64(grad_logp)
    gh = np.zeros_like(g) if grad_entropy is None else as_f64(grad_entropy)
    z = (h @ w.T) * float(inv_temperature)
    dz = _dz_rows(z, y, g, gh, inv_temperature)
    out = {"grad_hidden": dz @ w, "grad_w": dz.T @ h}
    if return_dz:
        out["dz"] = dz
    return out


def _dz_rows(z: np.ndarray, y: np.ndarray, g: np.ndarray, gh: np.ndarray, inv_temperature: float) -> np.ndarray:
    """dZ of a block of rows from their logits z [R, V] (module docstring):
    the two-pass log-softmax, the entropy, then the closed form."""
    m = z.max(axis=1)
    lse = m + np.log(np.exp(z - m[:, None]).sum(axis=1))
    logp_all = z - lse[:, None]
    p = np.exp(logp_all)
    ent = -(p * logp_all).sum(axis=1)
    onehot = np.zeros_like(z)
    onehot[np.arange(z.shape[0]), y] = 1.0
    return float(inv_temperature) * (g[:, None] * (onehot - p) - gh[:, None] * p * (logp_all + ent[:, None]))


def token_logprobs_bwd_rows(hidden, w_vocab, targets, grad_logp, grad_entropy=None,
                            inv_temperature: float = 1.0, vocab_rows=None, rows_per_block: int = 256):
    """The closed-form gradients of ``token_logprobs_bwd`` for problems too
    large to form Z whole: every row of grad_hidden, and grad_w at the
    vocabulary rows ``vocab_rows`` only (all rows when None).

    Rows t are independent up to dZ, so dZ is formed one block of rows at a
    time, each row over the full vocabulary (nothing in a row's log-softmax,
    entropy or dZ is blocked), and grad_hidden = dZ W per block. The columns
    vocab_rows of dZ are kept for all rows, and grad_w[vocab_rows] =
    dZ[:, vocab_rows]^T H is one product over all rows t.

    ``w_vocab`` may be a float64 array already (it is then used without a
    copy). Returns float64 ``grad_hidden`` [N, d] and ``grad_w`` [len(vocab_rows), d].
    """
    h = as_f64(hidden)
    w = as_f64(w_vocab)
    y = as_i64(targets)
    g = as_f64(grad_logp)
    gh = np.zeros_like(g) if grad_entropy is None else as_f64(grad_entropy)
    n, V = h.shape[0], w.shape[0]
    cols = np.arange(V) if vocab_rows is None else as_i64(vocab_rows)
    if n and (y.min() < 0 or y.max() >= V):
        raise ValueError("target out of range [0, V)")
    grad_hidden = np.empty_like(h)
    dz_cols = np.empty((n, cols.shape[0]))
    for r0 in range(0, n, rows_per_block):
        r1 = min(n, r0 + rows_per_block)
        z = (h[r0:r1] @ w.T) * float(inv_temperature)
        dz = _dz_rows(z, y[r0:r1], g[r0:r1], gh[r0:r1], inv_temperature)
        grad_hidden[r0:r1] = dz @ w
        dz_cols[r0:r1] = dz[:, cols]
    return {"grad_hidden": grad_hidden, "grad_w": dz_cols.T @ h}
