"""GPU masked GRPO loss (mc_grpo_masked_loss) vs the fp64 oracle, and the
whole chain forward -> filter -> loss -> backward vs the oracle chain.

Tolerances: the loss and the KL estimate within 2e-5 absolute (fp32 sums of
O(1) terms over up to ~1e5 tokens, normalised by Z); per-token gradients
within 1e-5 relative (plus 1e-6 of the largest gradient, where the surrogate
and KL terms cancel), except tokens whose ratio lies within 1e-5 (relative)
of a clip boundary,
where the fp32 and fp64 branch decisions may differ (the loss is continuous
there, its derivative is not)."""

import numpy as np
import pytest
import torch

import oracle
from gpu_util import TOL_GRAD, np_, rel_fro
from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def make(lens, seed=0, gap_std=0.3, mask_p=None, keep_p=0.7):
    g = torch.Generator().manual_seed(seed)
    cu = torch.zeros(len(lens) + 1, dtype=torch.int64)
    cu[1:] = torch.cumsum(torch.tensor(lens, dtype=torch.int64), 0)
    N = int(cu[-1])
    lp = -torch.rand(N, generator=g) * 6.0
    lb = (lp.double() + torch.randn(N, generator=g).double() * gap_std).float()
    mask = None if mask_p is None else (torch.rand(N, generator=g) < mask_p).to(torch.uint8)
    keep = (torch.rand(len(lens), generator=g) < keep_p).to(torch.uint8)
    adv = torch.randn(len(lens), generator=g)
    m = torch.ones(N, dtype=torch.uint8) if mask is None else mask
    n_tok = torch.tensor([int(m[cu[i]:cu[i + 1]].sum()) for i in range(len(lens))], dtype=torch.int32)
    return lp, lb, mask, cu, adv, keep, n_tok


def compare(lp, lb, mask, cu, adv, keep, n_tok, eps_low, eps_high, lr=None, beta=0.0):
    out = mc.grpo_masked_loss(lp.cuda(), lb.cuda(), None if mask is None else mask.cuda(), cu.cuda(), adv.cuda(),
                              keep.cuda(), n_tok.cuda(), eps_low, eps_high,
                              logp_ref=None if lr is None else lr.cuda(), beta=beta)
    torch.cuda.synchronize()
    ref = oracle.grpo_masked_loss(lp.numpy(), lb.numpy(), None if mask is None else mask.numpy(), cu.numpy(),
                                  adv.numpy(), keep.numpy(), float(np.float32(eps_low)), float(np.float32(eps_high)),
                                  logp_ref=None if lr is None else lr.numpy(), beta=float(np.float32(beta)))
    assert abs(float(out["loss"].item()) - ref["loss"]) <= 2e-5, (out["loss"].item(), ref["loss"])
    assert abs(float(out["kl"].item()) - ref["kl"]) <= 2e-5, (out["kl"].item(), ref["kl"])
    np.testing.assert_allclose(np_(out["seq_loss"]), ref["seq_loss"], atol=2e-6)
    rho = np.exp(lp.double().numpy() - lb.double().numpy())
    lo, hi = 1 - np.float32(eps_low), 1 + np.float32(eps_high)
    near = (np.abs(rho - lo) <= 1e-5 * lo) | (np.abs(rho - hi) <= 1e-5 * hi)
    g, gr = np_(out["grad_logp"]), ref["grad_logp"]
    ok = ~near
    # relative 1e-5, plus fp32 rounding of the two gradient terms where they cancel
    np.testing.assert_allclose(g[ok], gr[ok], rtol=1e-5, atol=1e-6 * float(np.abs(gr).max(initial=0.0)))
    seq = np.repeat(np.arange(len(adv)), np.diff(cu.numpy()))
    counted = keep.numpy()[seq].astype(bool) & (np.ones_like(seq, bool) if mask is None else mask.numpy().astype(bool))
    n_ref = int(ref["clipped"][counted].sum())
    assert abs(int(out["n_clipped"].item()) - n_ref) <= int(near[counted].sum())
    return out, ref


@pytest.mark.parametrize("eps", [(0.2, 0.2), (0.2, 0.28), (0.0, 0.0)])
def test_config_shaped(eps):
    lens = torch.randint(512, 8193, (32,), generator=torch.Generator().manual_seed(11)).tolist()
    compare(*make(lens, seed=1), *eps)


@pytest.mark.parametrize("beta", [0.0, 0.04, 1.0])
def test_kl_term(beta):
    lens = torch.randint(100, 3000, (24,), generator=torch.Generator().manual_seed(12)).tolist()
    lp, lb, mask, cu, adv, keep, n_tok = make(lens, seed=7, mask_p=0.85)
    lr = (lp.double() + torch.randn(lp.shape[0], generator=torch.Generator().manual_seed(3)).double() * 0.3).float()
    out, ref = compare(lp, lb, mask, cu, adv, keep, n_tok, 0.2, 0.28, lr=lr, beta=beta)
    assert ref["kl"] > 0


def test_ragged_masked_empty_and_unaligned():
    lens = [1, 0, 3, 5, 7, 0, 1, 130, 1023, 4, 9]
    lp, lb, mask, cu, adv, keep, n_tok = make(lens, seed=2, mask_p=0.6, keep_p=0.8)
    compare(lp, lb, mask, cu, adv, keep, n_tok, 0.2, 0.28)
    # 4-byte but not 16-byte aligned token arrays take the scalar path
    pad = lambda t: torch.cat([torch.zeros(1, dtype=t.dtype), t]).cuda()[1:]  # noqa: E731
    out = mc.grpo_masked_loss(pad(lp), pad(lb), mask.cuda(), cu.cuda(), adv.cuda(), keep.cuda(), n_tok.cuda(),
                              0.2, 0.28)
    ref = oracle.grpo_masked_loss(lp.numpy(), lb.numpy(), mask.numpy(), cu.numpy(), adv.numpy(), keep.numpy(),
                                  0.2, float(np.float32(0.28)))
    assert abs(out["loss"].item() - ref["loss"]) <= 2e-5


def test_all_dropped_and_on_policy():
    lp, lb, mask, cu, adv, keep, n_tok = make([40, 60, 25], seed=3)
    out = mc.grpo_masked_loss(lp.cuda(), lb.cuda(), None, cu.cuda(), adv.cuda(), torch.zeros(3, dtype=torch.uint8)
                              .cuda(), n_tok.cuda(), 0.2, 0.2)
    assert out["loss"].item() == 0.0 and not out["grad_logp"].any()
    out, ref = compare(lp, lp.clone(), None, cu, adv, torch.ones(3, dtype=torch.uint8), n_tok, 0.2, 0.2)
    assert int(out["n_clipped"].item()) == 0


def test_deterministic():
    args = make([300, 200, 700], seed=4)
    a = compare(*args, 0.2, 0.28)[0]
    b = compare(*args, 0.2, 0.28)[0]
    assert torch.equal(a["loss"], b["loss"]) and torch.equal(a["grad_logp"], b["grad_logp"])


def test_chain_forward_filter_loss_backward_tiny():
    """Tiny config end to end: every stage on the GPU vs every stage in the oracle."""
    wl = workloads.build(workloads.spec_for(1), "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    ref_fw = oracle.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    lb = torch.from_numpy(ref_fw["logp"] + wl.gap.double().numpy()).float()
    ref_flt0 = oracle.seq_ratio_filter(ref_fw["logp"], lb.numpy(), None, wl.cu_seqlens.numpy(), 1.0)
    a_sorted = np.sort(ref_flt0["abs_mean"])
    delta = float(0.5 * (a_sorted[3] + a_sorted[4]))  # a threshold well away from every statistic
    adv = torch.randn(wl.B, generator=torch.Generator().manual_seed(5))

    fw = mc.token_logprobs(h, w, y)
    flt = mc.seq_ratio_filter(fw["logp"], lb.cuda(), None, wl.cu_seqlens.cuda(), delta)
    loss = mc.grpo_masked_loss(fw["logp"], lb.cuda(), None, wl.cu_seqlens.cuda(), adv.cuda(), flt["keep"],
                               flt["n_tokens"], 0.2, 0.28)
    bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], loss["grad_logp"], None)
    torch.cuda.synchronize()

    ref_flt = oracle.seq_ratio_filter(ref_fw["logp"], lb.numpy(), None, wl.cu_seqlens.numpy(), float(np.float32(delta)))
    np.testing.assert_array_equal(np_(flt["keep"]), ref_flt["keep"])
    assert 0 < ref_flt["keep"].sum() < wl.B
    ref_loss = oracle.grpo_masked_loss(ref_fw["logp"], lb.numpy(), None, wl.cu_seqlens.numpy(), adv.numpy(),
                                       ref_flt["keep"], 0.2, float(np.float32(0.28)))
    assert abs(loss["loss"].item() - ref_loss["loss"]) <= 1e-4
    ref_bw = oracle.token_logprobs_bwd(wl.hidden, wl.w_vocab, wl.targets, ref_loss["grad_logp"])
    assert rel_fro(np_(bw["grad_hidden"].float()), ref_bw["grad_hidden"]) <= TOL_GRAD
    assert rel_fro(np_(bw["grad_w"]), ref_bw["grad_w"]) <= TOL_GRAD


def test_many_tiny_sequences():
    """100,003 sequences of 0-5 tokens: dozens of sequences per persistent
    CTA, and the last CTA's fixed-order sum over 100,003 per-sequence shares
    (not a multiple of the 4-share vector loads)."""
    lens = torch.randint(0, 6, (100_003,), generator=torch.Generator().manual_seed(13)).tolist()
    compare(*make(lens, seed=14, mask_p=0.8), 0.2, 0.28)
