"""Pins for the fp64 oracle of the log-prob / entropy forward and its backward.

Each pin checks the oracle against something other than itself: brute force in
plain Python floats, closed forms, invariants of the softmax, SciPy's
log_softmax / entropy, torch fp64 autograd, and central finite differences.
A plausible slip (a transposed operand, a wrong gather index, a dropped
temperature, an entropy sign, a dropped backward term) fails one of them.
"""

import math

import numpy as np
import pytest

import oracle
from oracle.logprobs import token_logprobs, token_logprobs_bwd, token_logprobs_bwd_rows

scipy_special = pytest.importorskip("scipy.special")


def _rand(rng, *shape, scale=1.0):
    return rng.standard_normal(shape) * scale


def _brute_force(h, w, y, inv_temp):
    """Plain Python loops: z_v = sum_k h_k w_vk, softmax, -sum p log p."""
    N, d = len(h), len(h[0])
    V = len(w)
    logp, ent = [], []
    for t in range(N):
        z = []
        for v in range(V):
            acc = 0.0
            for k in range(d):
                acc += h[t][k] * w[v][k]
            z.append(acc * inv_temp)
        denom = sum(math.exp(zv) for zv in z)
        p = [math.exp(zv) / denom for zv in z]
        logp.append(math.log(p[y[t]]))
        ent.append(-sum(pv * math.log(pv) for pv in p))
    return np.array(logp), np.array(ent)


@pytest.mark.parametrize("V", [2, 3, 8])
@pytest.mark.parametrize("inv_temp", [1.0, 1.0 / 0.9])
def test_brute_force_tiny_vocab(V, inv_temp):
    rng = np.random.default_rng(V)
    N, d = 5, 7  # N != V != d so a transposed operand cannot pass
    h, w = _rand(rng, N, d), _rand(rng, V, d, scale=0.5)
    y = rng.integers(0, V, N)
    out = token_logprobs(h, w, y, inv_temp)
    bl, be = _brute_force(h.tolist(), w.tolist(), y.tolist(), inv_temp)
    np.testing.assert_allclose(out["logp"], bl, rtol=0, atol=1e-12)
    np.testing.assert_allclose(out["entropy"], be, rtol=0, atol=1e-12)


def test_two_class_closed_form():
    """V = 2: logp_y = -log(1 + e^{z_o - z_y}); H is the binary entropy."""
    rng = np.random.default_rng(1)
    h, w = _rand(rng, 6, 4), _rand(rng, 2, 4)
    y = np.array([0, 1, 0, 1, 1, 0])
    out = token_logprobs(h, w, y)
    z = h @ w.T
    zy = z[np.arange(6), y]
    zo = z[np.arange(6), 1 - y]
    np.testing.assert_allclose(out["logp"], -np.log1p(np.exp(zo - zy)), atol=1e-13)
    p = 1.0 / (1.0 + np.exp(-(z[:, 0] - z[:, 1])))
    hb = -(p * np.log(p) + (1 - p) * np.log(1 - p))
    np.testing.assert_allclose(out["entropy"], hb, atol=1e-13)


def test_probabilities_sum_to_one():
    rng = np.random.default_rng(2)
    N, d, V = 3, 16, 37
    h, w = _rand(rng, N, d), _rand(rng, V, d, scale=0.3)
    total = np.zeros(N)
    for v in range(V):
        total += np.exp(token_logprobs(h, w, np.full(N, v))["logp"])
    np.testing.assert_allclose(total, 1.0, atol=1e-12)


def test_entropy_bounds_and_uniform_case():
    rng = np.random.default_rng(3)
    N, d, V = 16, 32, 100
    h = _rand(rng, N, d)
    out = token_logprobs(h, _rand(rng, V, d, scale=0.4), rng.integers(0, V, N))
    assert np.all(out["entropy"] >= -1e-12)
    assert np.all(out["entropy"] <= math.log(V) + 1e-12)
    # W = 0: every logit equal -> uniform softmax.
    u = token_logprobs(h, np.zeros((V, d)), rng.integers(0, V, N))
    np.testing.assert_allclose(u["logp"], -math.log(V), atol=1e-14)
    np.testing.assert_allclose(u["entropy"], math.log(V), atol=1e-13)
    np.testing.assert_allclose(u["lse"], math.log(V), atol=1e-13)


def test_one_hot_dominant_logit():
    """Margin 50 on one logit: H -> 0 and logp -> 0 at the peak, -50 elsewhere."""
    V, d = 10, 10
    h = np.eye(d)[:4] * 50.0
    w = np.eye(V, d)
    out = token_logprobs(h, w, np.array([0, 1, 2, 5]))
    np.testing.assert_allclose(out["logp"][:3], 0.0, atol=1e-19)
    np.testing.assert_allclose(out["logp"][3], -50.0, atol=1e-18)
    assert np.all(out["entropy"] < 1e-18)


def test_shift_invariance():
    """Adding c to every logit (an extra hidden column against a column of ones)
    changes lse by c and nothing else."""
    rng = np.random.default_rng(4)
    N, d, V = 8, 12, 50
    h, w = _rand(rng, N, d), _rand(rng, V, d, scale=0.5)
    y = rng.integers(0, V, N)
    c = 7.25
    a = token_logprobs(h, w, y)
    b = token_logprobs(np.hstack([h, np.full((N, 1), c)]), np.hstack([w, np.ones((V, 1))]), y)
    np.testing.assert_allclose(b["logp"], a["logp"], atol=1e-12)
    np.testing.assert_allclose(b["entropy"], a["entropy"], atol=1e-12)
    np.testing.assert_allclose(b["lse"], a["lse"] + c, atol=1e-12)


def test_temperature_equals_scaled_weights():
    rng = np.random.default_rng(5)
    N, d, V = 6, 8, 40
    h, w = _rand(rng, N, d), _rand(rng, V, d)
    y = rng.integers(0, V, N)
    a = token_logprobs(h, w, y, inv_temperature=2.0)
    b = token_logprobs(h, 2.0 * w, y)
    for k in ("logp", "entropy", "lse"):
        np.testing.assert_allclose(a[k], b[k], atol=1e-12)


def test_matches_scipy_on_tiny_config_shape():
    """Config-1 shape (N=256, d=512, V=4096) against scipy.special.log_softmax
    and scipy.special.entr, blocked rows and vocab included."""
    import torch

    from paper_2606_04847_gb300 import workloads

    wl = workloads.build(workloads.spec_for(1), "cpu")
    out = token_logprobs(wl.hidden, wl.w_vocab, wl.targets, rows_per_block=50,
                         vocab_per_block=1000)
    z = wl.hidden.to(torch.float64).numpy() @ wl.w_vocab.to(torch.float64).numpy().T
    ls = scipy_special.log_softmax(z, axis=1)
    y = wl.targets.numpy().astype(np.int64)
    np.testing.assert_allclose(out["logp"], ls[np.arange(wl.N), y], atol=1e-11)
    ent = scipy_special.entr(np.exp(ls)).sum(axis=1)
    np.testing.assert_allclose(out["entropy"], ent, atol=1e-10)
    np.testing.assert_allclose(out["lse"], scipy_special.logsumexp(z, axis=1), atol=1e-11)


def test_target_range_is_an_error():
    with pytest.raises(ValueError):
        token_logprobs(np.ones((2, 4)), np.ones((3, 4)), np.array([0, 3]))
    with pytest.raises(ValueError):
        token_logprobs(np.ones((2, 4)), np.ones((3, 4)), np.array([-1, 0]))


def test_shard_states_recombine_to_the_full_vocabulary():
    """States of disjoint vocabulary shards, combined by rescaling to a common
    max, give the full-vocabulary lse, entropy and target logit."""
    from oracle.logprobs import logprob_state

    rng = np.random.default_rng(9)
    N, d, V = 7, 16, 50
    h, w = _rand(rng, N, d), _rand(rng, V, d, scale=0.6)
    y = rng.integers(0, V, N)
    full = token_logprobs(h, w, y)
    bounds = [0, 13, 14, 40, 50]  # includes a one-column shard
    st = [logprob_state(h, w[a:b], y, a) for a, b in zip(bounds[:-1], bounds[1:])]
    M = np.max([s[:, 0] for s in st], axis=0)
    S = sum(s[:, 1] * np.exp(s[:, 0] - M) for s in st)
    T = sum(np.exp(s[:, 0] - M) * (s[:, 2] + (s[:, 0] - M) * s[:, 1]) for s in st)
    zy = np.max([s[:, 3] for s in st], axis=0)
    np.testing.assert_allclose(M + np.log(S), full["lse"], atol=1e-12)
    np.testing.assert_allclose(np.log(S) - T / S, full["entropy"], atol=1e-12)
    np.testing.assert_allclose(zy - (M + np.log(S)), full["logp"], atol=1e-12)
    # exactly one shard owns each target
    owners = sum(np.isfinite(s[:, 3]).astype(int) for s in st)
    np.testing.assert_array_equal(owners, 1)
    for s in st:
        assert np.all(s[:, 1] >= 1.0) and np.all(s[:, 2] <= 0.0)


# ---------------------------------------------------------------- backward


def _loss(h, w, y, g, gh, inv_temp):
    out = token_logprobs(h, w, y, inv_temp)
    return float((g * out["logp"]).sum() + (gh * out["entropy"]).sum())


@pytest.mark.parametrize("inv_temp", [1.0, 1.0 / 0.9])
def test_backward_central_differences(inv_temp):
    rng = np.random.default_rng(6)
    N, d, V = 4, 8, 16
    h, w = _rand(rng, N, d), _rand(rng, V, d, scale=0.7)
    y = rng.integers(0, V, N)
    g, gh = _rand(rng, N), _rand(rng, N)
    out = token_logprobs_bwd(h, w, y, g, gh, inv_temp)
    eps = 1e-6
    for arr, grad in ((h, out["grad_hidden"]), (w, out["grad_w"])):
        fd = np.zeros_like(arr)
        for idx in np.ndindex(arr.shape):
            old = arr[idx]
            arr[idx] = old + eps
            lp = _loss(h, w, y, g, gh, inv_temp)
            arr[idx] = old - eps
            lm = _loss(h, w, y, g, gh, inv_temp)
            arr[idx] = old
            fd[idx] = (lp - lm) / (2 * eps)
        err = np.linalg.norm(fd - grad) / np.linalg.norm(grad)
        assert err < 1e-7, err


def test_backward_matches_torch_autograd_fp64():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(7)
    N, d, V = 9, 24, 70
    h, w = _rand(rng, N, d), _rand(rng, V, d, scale=0.5)
    y = rng.integers(0, V, N)
    g, gh = _rand(rng, N), _rand(rng, N)
    inv_temp = 1.3
    th = torch.tensor(h, requires_grad=True)
    tw = torch.tensor(w, requires_grad=True)
    ls = torch.log_softmax((th @ tw.T) * inv_temp, dim=1)
    logp = ls[torch.arange(N), torch.tensor(y)]
    ent = -(ls.exp() * ls).sum(dim=1)
    ((torch.tensor(g) * logp).sum() + (torch.tensor(gh) * ent).sum()).backward()
    out = token_logprobs_bwd(h, w, y, g, gh, inv_temp)
    np.testing.assert_allclose(out["grad_hidden"], th.grad.numpy(), atol=1e-12)
    np.testing.assert_allclose(out["grad_w"], tw.grad.numpy(), atol=1e-12)


def test_backward_invariants():
    rng = np.random.default_rng(8)
    N, d, V = 6, 10, 33
    h, w = _rand(rng, N, d), _rand(rng, V, d)
    y = rng.integers(0, V, N)
    out = token_logprobs_bwd(h, w, y, _rand(rng, N), _rand(rng, N), 0.8, return_dz=True)
    # Each softmax-gradient row sums to zero (both terms are orthogonal to 1).
    np.testing.assert_allclose(out["dz"].sum(axis=1), 0.0, atol=1e-13)
    z0 = token_logprobs_bwd(h, w, y, np.zeros(N), None)
    assert not np.any(z0["grad_hidden"]) and not np.any(z0["grad_w"])


def test_backward_rows_matches_torch_autograd_fp64():
    """The row-blocked variant used at full problem sizes (ragged last block,
    an unsorted subset of vocabulary rows with repeats) against torch fp64
    autograd of the log-softmax and entropy."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(9)
    N, d, V = 11, 16, 45
    h, w = _rand(rng, N, d), _rand(rng, V, d, scale=0.6)
    y = rng.integers(0, V, N)
    g, gh = _rand(rng, N), _rand(rng, N)
    inv_temp = 1.0 / 0.9
    th = torch.tensor(h, requires_grad=True)
    tw = torch.tensor(w, requires_grad=True)
    ls = torch.log_softmax((th @ tw.T) * inv_temp, dim=1)
    logp = ls[torch.arange(N), torch.tensor(y)]
    ent = -(ls.exp() * ls).sum(dim=1)
    ((torch.tensor(g) * logp).sum() + (torch.tensor(gh) * ent).sum()).backward()
    cols = np.array([44, 0, int(y[3]), 17, 17, 30])
    out = token_logprobs_bwd_rows(h, w, y, g, gh, inv_temp, vocab_rows=cols, rows_per_block=4)
    np.testing.assert_allclose(out["grad_hidden"], th.grad.numpy(), atol=1e-12)
    np.testing.assert_allclose(out["grad_w"], tw.grad.numpy()[cols], atol=1e-12)
    # All vocabulary rows: each dZ row sums to zero, so grad_w sums to zero over v.
    full = token_logprobs_bwd_rows(h, w, y, g, None, inv_temp, rows_per_block=3)
    assert full["grad_w"].shape == (V, d)
    np.testing.assert_allclose(full["grad_w"].sum(axis=0), 0.0, atol=1e-12)


def test_oracle_package_exports():
    assert callable(oracle.token_logprobs) and callable(oracle.seq_ratio_filter)
