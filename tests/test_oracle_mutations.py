"""Planted mistakes, on the CPU: each plausible slip is applied as a text
patch to a copy of one oracle module, and the patched copy must fail at least
one of the checks below, while the unpatched module passes them all. The
checks are written here without the oracle's code: brute force in plain
Python floats, closed forms, the paper's worked example (ρ = [10, 0.1],
§4.5.2), hand-computed cases and central finite differences. This is the
evidence that the oracle's pins catch slips of these kinds.
"""

import math
import os
import types

import numpy as np
import pytest

ORACLE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle")


def load(module, patch=None):
    """A fresh copy of oracle/<module>.py, optionally with one text patch
    (old, new) applied exactly once."""
    path = os.path.join(ORACLE, module + ".py")
    src = open(path).read()
    if patch is not None:
        old, new = patch
        assert src.count(old) == 1, f"patch does not apply exactly once: {old!r}"
        src = src.replace(old, new)
    mod = types.ModuleType(f"oracle._copy_of_{module}")
    mod.__package__ = "oracle"  # relative imports resolve to the real package
    exec(compile(src, path, "exec"), mod.__dict__)
    return mod


def fails(check, mod):
    try:
        check(mod)
    except (AssertionError, ValueError, IndexError, FloatingPointError):
        return True
    return False


# ------------------------------------------------------------------ log-probs


def _softmax_row(z):
    m = max(z)
    e = [math.exp(v - m) for v in z]
    s = sum(e)
    return [v / s for v in e], m + math.log(s)


def _brute(h, w, y, inv_temp):
    out = {"logp": [], "entropy": [], "lse": []}
    for t in range(len(h)):
        z = [sum(h[t][k] * w[v][k] for k in range(len(h[t]))) * inv_temp for v in range(len(w))]
        p, lse = _softmax_row(z)
        out["logp"].append(z[y[t]] - lse)
        out["entropy"].append(-sum(q * math.log(q) for q in p if q > 0))
        out["lse"].append(lse)
    return out


def check_forward(mod):
    rng = np.random.default_rng(0)
    for V in (2, 3, 8):
        for inv_temp in (1.0, 1.0 / 0.9):
            h = rng.standard_normal((5, 4))
            w = rng.standard_normal((V, 4))
            y = rng.integers(0, V, 5)
            got = mod.token_logprobs(h, w, y, inv_temp)
            ref = _brute(h.tolist(), w.tolist(), y.tolist(), inv_temp)
            for k in ("logp", "entropy", "lse"):
                assert np.allclose(got[k], ref[k], atol=1e-9), k
    h = rng.standard_normal((3, 4))
    got = mod.token_logprobs(h, np.zeros((7, 4)), np.array([0, 3, 6]))
    assert np.allclose(got["logp"], -math.log(7)) and np.allclose(got["entropy"], math.log(7))


def _brute_loss(h, w, y, g, gh, inv_temp):
    r = _brute(h, w, y, inv_temp)
    return sum(g[t] * r["logp"][t] + gh[t] * r["entropy"][t] for t in range(len(h)))


def check_backward(mod):
    rng = np.random.default_rng(1)
    N, d, V, inv_temp = 3, 4, 6, 1.0 / 0.9
    h, w = rng.standard_normal((N, d)), rng.standard_normal((V, d))
    y, g, gh = rng.integers(0, V, N), rng.standard_normal(N), rng.standard_normal(N)
    got = mod.token_logprobs_bwd(h, w, y, g, gh, inv_temp)
    eps = 1e-6
    for name, x, grad in (("grad_hidden", h, got["grad_hidden"]), ("grad_w", w, got["grad_w"])):
        fd = np.zeros_like(x)
        for idx in np.ndindex(x.shape):
            xp, xm = x.copy(), x.copy()
            xp[idx] += eps
            xm[idx] -= eps
            args_p = (xp, w) if name == "grad_hidden" else (h, xp)
            args_m = (xm, w) if name == "grad_hidden" else (h, xm)
            fd[idx] = (_brute_loss(args_p[0].tolist(), args_p[1].tolist(), y.tolist(), g, gh, inv_temp)
                       - _brute_loss(args_m[0].tolist(), args_m[1].tolist(), y.tolist(), g, gh, inv_temp)) / (2 * eps)
        assert np.allclose(grad, fd, rtol=1e-6, atol=1e-8), name


LOGPROB_SLIPS = [
    ("ent = lse - (p * z).sum(axis=1)", "ent = (p * z).sum(axis=1) - lse"),          # entropy sign
    ("        z *= float(inv_temperature)\n", "        z *= 1.0\n"),                 # dropped temperature
    ("logp = z[rows, y] - lse", "logp = z[rows, y - 1] - lse"),                      # wrong gather index
    ("lse = m + np.log(np.exp(z - m[:, None]).sum(axis=1))\n    rows",
     "lse = np.log(np.exp(z - m[:, None]).sum(axis=1))\n    rows"),                    # dropped max shift
]
BACKWARD_SLIPS = [
    ("(g[:, None] * (onehot - p) - gh[:, None] * p * (logp_all + ent[:, None]))",
     "(g[:, None] * (onehot - p))"),                                                  # dropped entropy term
    ("return float(inv_temperature) * (", "return 1.0 * ("),                          # dropped temperature
    ("(g[:, None] * (onehot - p)", "(g[:, None] * (p - onehot)"),                    # sign of the softmax term
    ("(logp_all + ent[:, None])", "(logp_all - ent[:, None])"),                      # sign inside the entropy term
    ('"grad_w": dz.T @ h', '"grad_w": dz.T @ (h * 0.5)'),                            # a stray factor on one GEMM
]
# Slips in the row-blocked variant used at full problem sizes.
BACKWARD_ROWS_SLIPS = [
    ("dz_cols[r0:r1] = dz[:, cols]", "dz_cols[r0:r1] = dz[:, cols - 1]"),            # wrong vocabulary column
    ("r1 = min(n, r0 + rows_per_block)\n        z = (h[r0:r1] @ w.T)",
     "r1 = min(n, r0 + rows_per_block)\n        z = (h[r0:r1] @ w.T) * 0 + (h[r0:r1] @ w.T)[:, ::-1]"),
                                                                                      # reversed vocabulary order
    ('"grad_w": dz_cols.T @ h}', '"grad_w": dz_cols.T @ h[::-1]}'),                 # rows of H misaligned with dZ
    ("grad_hidden[r0:r1] = dz @ w\n", "grad_hidden[r0:r1] = dz @ w * float(inv_temperature)\n"),
                                                                                      # temperature applied twice
    ("for r0 in range(0, n, rows_per_block):\n        r1 = min(n, r0 + rows_per_block)\n        z = (h",
     "for r0 in range(0, n - 1, rows_per_block):\n        r1 = min(n, r0 + rows_per_block)\n        z = (h"),
                                                                                      # last block dropped
]


def check_backward_rows(mod):
    """Row-blocked gradients (ragged last block, unsorted vocabulary rows)
    against central differences of the brute-force loss."""
    rng = np.random.default_rng(2)
    N, d, V, inv_temp = 5, 4, 6, 1.0 / 0.9
    h, w = rng.standard_normal((N, d)), rng.standard_normal((V, d))
    y, g, gh = rng.integers(0, V, N), rng.standard_normal(N), rng.standard_normal(N)
    cols = np.array([5, 0, 3])
    np.seterr(all="raise")
    try:
        got = mod.token_logprobs_bwd_rows(h, w, y, g, gh, inv_temp, vocab_rows=cols, rows_per_block=2)
    finally:
        np.seterr(all="warn")
    eps = 1e-6

    def fd(which, idx):
        xp, xm = (h.copy(), w.copy()), (h.copy(), w.copy())
        xp[which][idx] += eps
        xm[which][idx] -= eps
        lp = _brute_loss(xp[0].tolist(), xp[1].tolist(), y.tolist(), g, gh, inv_temp)
        lm = _brute_loss(xm[0].tolist(), xm[1].tolist(), y.tolist(), g, gh, inv_temp)
        return (lp - lm) / (2 * eps)

    want_h = np.array([[fd(0, (t, k)) for k in range(d)] for t in range(N)])
    want_w = np.array([[fd(1, (v, k)) for k in range(d)] for v in cols])
    assert np.allclose(got["grad_hidden"], want_h, rtol=1e-6, atol=1e-8), "grad_hidden"
    assert np.allclose(got["grad_w"], want_w, rtol=1e-6, atol=1e-8), "grad_w rows"


def test_unpatched_log_prob_oracle_passes():
    mod = load("logprobs")
    check_forward(mod)
    check_backward(mod)
    check_backward_rows(mod)


@pytest.mark.parametrize("patch", LOGPROB_SLIPS, ids=lambda p: p[1][:40])
def test_forward_slip_is_caught(patch):
    assert fails(check_forward, load("logprobs", patch))


@pytest.mark.parametrize("patch", BACKWARD_SLIPS, ids=lambda p: p[1][:40])
def test_backward_slip_is_caught(patch):
    assert fails(check_backward, load("logprobs", patch))


@pytest.mark.parametrize("patch", BACKWARD_ROWS_SLIPS, ids=lambda p: p[1][:40])
def test_backward_rows_slip_is_caught(patch):
    assert fails(check_backward_rows, load("logprobs", patch))


# ------------------------------------------------------------------ filter


def check_filter(mod):
    # the paper's worked example: rho = [10, 0.1]
    lp = np.log(np.array([10.0, 0.1]))
    r = mod.seq_ratio_filter(lp, np.zeros(2), None, np.array([0, 2]), math.log(10), math.log(10))
    assert abs(r["signed_mean"][0]) < 1e-12 and abs(r["abs_mean"][0] - math.log(10)) < 1e-12
    assert r["keep"][0] == 1                      # A = delta is kept (Eq. 21: <=)
    assert np.allclose(r["token_ratio"], [10.0, 0.1])
    r = mod.seq_ratio_filter(lp, np.zeros(2), None, np.array([0, 2]), math.log(10) - 1e-9, -1.0)
    assert r["keep"][0] == 0
    # a constant gap g: S = g, A = |g|; masked tokens do not count
    lp = np.array([0.3, 0.3, 5.0, 0.3])
    mask = np.array([1, 1, 0, 1], dtype=np.uint8)
    r = mod.seq_ratio_filter(lp, np.zeros(4), mask, np.array([0, 4]), 0.5, 0.5)
    assert r["n_tokens"][0] == 3
    assert abs(r["signed_mean"][0] - 0.3) < 1e-12 and abs(r["abs_mean"][0] - 0.3) < 1e-12
    assert list(r["token_keep"]) == [1, 1, 0, 1]
    r = mod.seq_ratio_filter(-lp, np.zeros(4), mask, np.array([0, 4]), 0.5, 0.5)
    assert abs(r["signed_mean"][0] + 0.3) < 1e-12 and abs(r["abs_mean"][0] - 0.3) < 1e-12


FILTER_SLIPS = [
    ("A[i] = np.abs(sel).sum() / L[i]", "A[i] = np.abs(sel.sum()) / L[i]"),          # |sum| for sum|.|
    ("keep[i] = 1 if A[i] <= delta else 0", "keep[i] = 1 if A[i] < delta else 0"),   # < for <=
    ("log_rho = lp - lb", "log_rho = lb - lp"),                                      # ratio direction
    ("sel = log_rho[sl][mask[sl]]", "sel = log_rho[sl]"),                            # mask ignored
    ("token_keep[sl] = keep[i] & mask[sl]", "token_keep[sl] = keep[i]"),             # token_keep ignores the mask
    ("keep[i] = 1 if A[i] <= delta else 0", "keep[i] = 1 if abs(S[i]) <= delta else 0"),  # Vanilla for MirrorPop
]


def test_unpatched_filter_oracle_passes():
    check_filter(load("filter"))


@pytest.mark.parametrize("patch", FILTER_SLIPS, ids=lambda p: p[1][:40])
def test_filter_slip_is_caught(patch):
    assert fails(check_filter, load("filter", patch))


# ------------------------------------------------------------------ GRPO loss


def _loss_by_hand(lp, lb, lr, A, M, eps_low, eps_high, beta):
    """One response of masked tokens, Eq. 17 written out in Python floats."""
    Z = M * len(lp)
    total = 0.0
    for a, b, c in zip(lp, lb, lr):
        rho = math.exp(a - b)
        s = min(rho * A, min(max(rho, 1 - eps_low), 1 + eps_high) * A)
        k = math.exp(c - a) - (c - a) - 1
        total += M * (-s + beta * k)
    return total / Z if Z else 0.0


def check_loss(mod):
    lp = np.array([-0.1, -2.0, -0.5])
    lb = np.array([-0.4, -1.0, -0.5])
    lr = np.array([-0.2, -1.7, -0.9])
    cu = np.array([0, 3])
    for A in (1.3, -0.7):
        for eps_low, eps_high in ((0.2, 0.2), (0.1, 0.3)):
            r = mod.grpo_masked_loss(lp, lb, None, cu, np.array([A]), np.array([1]), eps_low, eps_high,
                                     logp_ref=lr, beta=0.04)
            assert abs(r["loss"] - _loss_by_hand(lp, lb, lr, A, 1, eps_low, eps_high, 0.04)) < 1e-12
            # dL/dlogp by central differences of the hand-written loss
            for t in range(3):
                e = 1e-6
                up, dn = lp.copy(), lp.copy()
                up[t] += e
                dn[t] -= e
                fd = (_loss_by_hand(up, lb, lr, A, 1, eps_low, eps_high, 0.04)
                      - _loss_by_hand(dn, lb, lr, A, 1, eps_low, eps_high, 0.04)) / (2 * e)
                assert abs(r["grad_logp"][t] - fd) < 1e-6, (t, r["grad_logp"][t], fd)
    # a dropped response counts in neither the sum nor the normaliser
    r = mod.grpo_masked_loss(np.concatenate([lp, lp]), np.concatenate([lb, lb]), None, np.array([0, 3, 6]),
                             np.array([1.3, 5.0]), np.array([1, 0]), 0.2, 0.2)
    assert abs(r["loss"] - _loss_by_hand(lp, lb, lp, 1.3, 1, 0.2, 0.2, 0.0)) < 1e-12
    assert not r["grad_logp"][3:].any()


LOSS_SLIPS = [
    ("s = min(unclipped, clipped_term)", "s = max(unclipped, clipped_term)"),         # max for min
    ("Z = float((M * L).sum())", "Z = float(L.sum())"),                               # sum L_i for sum M_i L_i
    ("seq_loss[i] -= s * M[i] / Z", "seq_loss[i] -= s / Z"),                          # dropped M_i
    ("np.clip(rho, 1.0 - eps_low, 1.0 + eps_high)", "np.clip(rho, 1.0 - eps_high, 1.0 + eps_low)"),  # swapped eps
    ("clipped[t] = True\n            elif M[i] != 0.0:", "clipped[t] = True\n            if M[i] != 0.0:"),  # grad through the clip
    ("k = np.exp(r) - r - 1.0", "k = np.exp(r) - r"),                                 # KL estimate off by one
    ("(1.0 - np.exp(r))", "(np.exp(r) - 1.0)"),                                       # KL gradient sign
]


def test_unpatched_loss_oracle_passes():
    check_loss(load("grpo"))


@pytest.mark.parametrize("patch", LOSS_SLIPS, ids=lambda p: p[1][:40])
def test_loss_slip_is_caught(patch):
    assert fails(check_loss, load("grpo", patch))


# ------------------------------------------------------------------ reward / advantage


def check_advantage(mod):
    s = np.array([[0.2, 0.9, 0.5], [0.7, 0.1, 0.3], [0.0, 0.0, 0.0]])
    ok = np.array([[0, 1, 0], [1, 0, 0], [0, 0, 1]], dtype=bool)
    nt = np.array([3, 3, 3])
    # alpha = 1: the first-turn score; alpha = 0: the best score (Eq. 9), no bonus
    assert np.allclose(mod.prime_echo_reward(s, ok, nt, 1.0, 0.0, 0.0), [0.2, 0.7, 0.0])
    assert np.allclose(mod.prime_echo_reward(s, ok, nt, 0.0, 0.0, 0.0), [0.9, 0.7, 0.0])
    # Eq. 10: beta2 only for a second-turn success after a first-turn failure
    ok4 = np.array([[0, 1, 0], [1, 0, 0], [0, 0, 1], [1, 1, 0]], dtype=bool)
    assert np.allclose(mod.prime_echo_reward(np.zeros((4, 3)), ok4, np.full(4, 3), 0.5, 0.5, 0.2),
                       [0.2, 0.5, 0.0, 0.5])
    # Eq. 12 with the sample std: zero mean and sum of squares G - 1 per group
    R = np.array([0.3, 1.2, -0.4, 2.0, 0.9, 0.1])
    A = mod.group_advantage(R, 3, 0.0)
    for g0 in (0, 3):
        assert abs(A[g0:g0 + 3].sum()) < 1e-12 and abs((A[g0:g0 + 3] ** 2).sum() - 2.0) < 1e-12


ADVANTAGE_SLIPS = [
    ("alpha * s[i, 0] + (1.0 - alpha) * best", "(1.0 - alpha) * s[i, 0] + alpha * best"),  # weights swapped
    ("(not first_ok and second_ok)", "second_ok"),                                       # beta2 after a first success
    ("/ (group_size - 1))", "/ group_size)"),                                            # population std
]


def test_unpatched_advantage_oracle_passes():
    check_advantage(load("advantage"))


@pytest.mark.parametrize("patch", ADVANTAGE_SLIPS, ids=lambda p: p[1][:40])
def test_advantage_slip_is_caught(patch):
    assert fails(check_advantage, load("advantage", patch))
