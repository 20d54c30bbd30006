"""Parity at the configured full sizes, in the launch configuration bench.py
times (whole batches through the C ABI, default workspaces).

* forward: every row runs on the GPU; a seeded sample of rows (including the
  first and last, i.e. the ragged last row block) is recomputed by the fp64
  oracle one row at a time.
* filter: the full batch of sequences, filter-only parity (both sides get the
  same fp32 log-prob arrays with the config's lengths, gaps and masks).
* backward (9B-class fwd+bwd): grad_hidden rows depend on their own row only,
  so sampled rows are checked against the oracle; grad_w sums over all kept
  rows, so it is checked through identities that hold at any size:
  <grad_hidden, H> = <grad_w, W> (both equal sum_{t,v} dZ[t,v] h_t.w_v) and
  sum_v grad_w[v, :] = 0 (each softmax-gradient row sums to zero).
"""

import numpy as np
import pytest
import torch

import oracle
from gpu_util import (MASK_BAND, TOL_ENT, TOL_GRAD, TOL_LOGP, TOL_RATIO, assert_close_abs, assert_close_rel,
                      assert_masks_match, np_, rel_fro)
from paper_2606_04847_gb300 import mc, workloads

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def sample_rows(n, k=16, seed=0):
    g = np.random.default_rng(seed)
    rows = set(g.choice(n, size=min(k - 2, n), replace=False).tolist())
    rows.update([0, n - 1])
    return np.array(sorted(rows))


@pytest.fixture(scope="module")
def w_cpu_cache():
    return {}


@pytest.mark.parametrize("config", [2, 3, 4, 5])
def test_forward_full_size(config, w_cpu_cache):
    spec = workloads.spec_for(config)
    wl = workloads.build(spec, "cuda")
    out = mc.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    torch.cuda.synchronize()
    rows = sample_rows(wl.N, seed=config)
    ridx = torch.from_numpy(rows).cuda()
    h = wl.hidden[ridx].cpu()
    y = wl.targets[ridx].cpu()
    w = wl.w_vocab.cpu()
    ref = oracle.token_logprobs(h, w, y, spec.inv_temperature)
    assert_close_abs(np_(out["logp"][ridx]), ref["logp"], TOL_LOGP, f"config {config} logp")
    assert_close_abs(np_(out["entropy"][ridx]), ref["entropy"], TOL_ENT, f"config {config} entropy")
    assert_close_abs(np_(out["lse"][ridx]), ref["lse"], TOL_LOGP, f"config {config} lse")
    assert torch.isfinite(out["logp"]).all() and torch.isfinite(out["entropy"]).all()


@pytest.mark.parametrize("config", [1, 2, 3, 4])
@pytest.mark.parametrize("cancel", [False, True])
def test_filter_full_size(config, cancel):
    spec = workloads.spec_for(config, d=64, V=128)  # shapes of the token arrays only
    wl = workloads.build(spec, "cpu")
    g = torch.Generator().manual_seed(config)
    lp = -torch.empty(wl.N).exponential_(0.5, generator=g)  # log-prob-like values
    gap = workloads.cancellation_gap(wl) if cancel else wl.gap
    lb = (lp.double() + gap.double()).float()
    mask = wl.loss_mask
    delta = spec.delta
    out = mc.seq_ratio_filter(lp.cuda(), lb.cuda(), mask.cuda(), wl.cu_seqlens.cuda(), delta, delta)
    ref = oracle.seq_ratio_filter(lp.numpy(), lb.numpy(), mask.numpy(), wl.cu_seqlens.numpy(),
                                  float(np.float32(delta)), float(np.float32(delta)))
    np.testing.assert_array_equal(np_(out["n_tokens"]), ref["n_tokens"])
    assert_close_rel(np.exp(np_(out["signed_mean"])), np.exp(ref["signed_mean"]), TOL_RATIO, "e^S")
    assert_close_rel(np.exp(np_(out["abs_mean"])), np.exp(ref["abs_mean"]), TOL_RATIO, "e^A")
    assert_close_rel(np_(out["token_ratio"]), ref["token_ratio"], TOL_RATIO, "rho_t")
    assert_masks_match(np_(out["keep"]), ref["keep"], ref["abs_mean"], delta, MASK_BAND, "keep")
    assert_masks_match(np_(out["keep_vanilla"]), ref["keep_vanilla"], np.abs(ref["signed_mean"]), delta,
                       MASK_BAND, "keep_vanilla")


def test_filter_full_size_first_turn_mask():
    """27B-class multi-turn batch with the paper's first-turn-only loss mask
    (only the first turn's response tokens count)."""
    spec = workloads.spec_for(4, d=64, V=128)
    wl = workloads.build(spec, "cpu", first_turn_only=True)
    g = torch.Generator().manual_seed(44)
    lp = -torch.empty(wl.N).exponential_(0.5, generator=g)
    lb = (lp.double() + wl.gap.double()).float()
    mask, delta = wl.loss_mask, spec.delta
    out = mc.seq_ratio_filter(lp.cuda(), lb.cuda(), mask.cuda(), wl.cu_seqlens.cuda(), delta, delta)
    ref = oracle.seq_ratio_filter(lp.numpy(), lb.numpy(), mask.numpy(), wl.cu_seqlens.numpy(),
                                  float(np.float32(delta)), float(np.float32(delta)))
    np.testing.assert_array_equal(np_(out["n_tokens"]), ref["n_tokens"])
    assert_close_rel(np.exp(np_(out["abs_mean"])), np.exp(ref["abs_mean"]), TOL_RATIO, "e^A")
    assert_masks_match(np_(out["keep"]), ref["keep"], ref["abs_mean"], delta, MASK_BAND, "keep")
    seq = np.repeat(np.arange(wl.B), np.diff(wl.cu_seqlens.numpy()))
    np.testing.assert_array_equal(np_(out["token_keep"]).astype(bool),
                                  np_(out["keep"]).astype(bool)[seq] & mask.numpy().astype(bool))


@pytest.mark.parametrize("config,first_turn", [(4, False), (4, True), (5, False)])
def test_loss_full_size(config, first_turn):
    """Masked GRPO loss with the beta * KL term (Eq. 17) on the configuration's
    sequence lengths and loss mask (config 4: multi-turn, prompt tokens masked,
    every turn or the first turn only), keep-mask from the filter, asymmetric
    clip."""
    spec = workloads.spec_for(config, d=64, V=128)  # shapes of the token arrays only
    wl = workloads.build(spec, "cpu", first_turn_only=first_turn)
    g = torch.Generator().manual_seed(40 + config)
    lp = -torch.empty(wl.N).exponential_(0.5, generator=g)
    lb = (lp.double() + wl.gap.double()).float()
    lr = (lp.double() + torch.randn(wl.N, generator=g).double() * 0.1).float()
    adv = torch.randn(wl.B, generator=g)
    mask = wl.loss_mask
    flt = mc.seq_ratio_filter(lp.cuda(), lb.cuda(), mask.cuda(), wl.cu_seqlens.cuda(), spec.delta)
    out = mc.grpo_masked_loss(lp.cuda(), lb.cuda(), mask.cuda(), wl.cu_seqlens.cuda(), adv.cuda(), flt["keep"],
                              flt["n_tokens"], 0.2, 0.28, logp_ref=lr.cuda(), beta=0.04)
    torch.cuda.synchronize()
    keep = np_(flt["keep"])
    ref = oracle.grpo_masked_loss(lp.numpy(), lb.numpy(), mask.numpy(), wl.cu_seqlens.numpy(), adv.numpy(), keep,
                                  float(np.float32(0.2)), float(np.float32(0.28)), logp_ref=lr.numpy(),
                                  beta=float(np.float32(0.04)))
    assert abs(out["loss"].item() - ref["loss"]) <= 2e-5, (out["loss"].item(), ref["loss"])
    assert abs(out["kl"].item() - ref["kl"]) <= 2e-5, (out["kl"].item(), ref["kl"])
    gr = ref["grad_logp"]
    rho = np.exp(lp.double().numpy() - lb.double().numpy())
    near = (np.abs(rho - 0.8) <= 1e-5) | (np.abs(rho - 1.28) <= 1.28e-5)
    np.testing.assert_allclose(np_(out["grad_logp"])[~near], gr[~near], rtol=1e-5,
                               atol=1e-6 * float(np.abs(gr).max(initial=0.0)))


def test_backward_full_size_9b():
    spec = workloads.spec_for(5)
    wl = workloads.build(spec, "cuda")
    h, w, y = wl.hidden, wl.w_vocab, wl.targets
    fw = mc.token_logprobs(h, w, y)
    # A seeded per-sequence keep mask (every third sequence dropped) given to both sides.
    keep_seq = torch.ones(wl.B, dtype=torch.uint8)
    keep_seq[::3] = 0
    lens = torch.tensor(wl.seq_lens, dtype=torch.int64)
    row_keep = torch.repeat_interleave(keep_seq, lens).cuda()
    bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], wl.advantages, None, row_keep=row_keep)
    torch.cuda.synchronize()
    gh, gw = bw["grad_hidden"], bw["grad_w"]
    assert torch.isfinite(gw).all()

    # Sampled grad_hidden rows (each depends on its own row only).
    rows = sample_rows(wl.N, k=12, seed=5)
    ridx = torch.from_numpy(rows).cuda()
    g_rows = (wl.advantages[ridx] * row_keep[ridx].float()).cpu()
    ref = oracle.token_logprobs_bwd(h[ridx].cpu(), w.cpu(), y[ridx].cpu(), g_rows)
    got = np_(gh[ridx].float())
    for i, r in enumerate(rows):
        if g_rows[i] == 0:
            assert not got[i].any(), f"dropped row {r} has a gradient"
        else:
            e = rel_fro(got[i], ref["grad_hidden"][i])
            assert e <= TOL_GRAD, f"row {r}: rel err {e:.3e}"

    # <grad_hidden, H> = <grad_w, W>, in fp64 on the GPU.
    # Tolerance: 1e-2 relative plus the bf16 rounding of grad_hidden itself
    # (std ~ 2^-9 / sqrt(3) * ||grad_hidden||_F * rms(H), rms(H) ~ 1).
    lhs = (gh.double() * h.double()).sum().item()
    rhs = (gw.double() * w.double()).sum().item()
    fro = gh.double().norm().item()
    assert abs(lhs - rhs) <= TOL_GRAD * max(abs(lhs), abs(rhs)) + 0.02 * fro, (lhs, rhs, fro)
    # sum over the vocabulary of grad_w is zero up to rounding (relative to the column scale).
    col = gw.double().sum(dim=0)
    scale = gw.double().abs().sum(dim=0)
    assert (col.abs() <= 1e-3 * scale + 1e-6).all()


def test_full_size_step_is_bitwise_reproducible():
    """Two runs of the 9B-class forward + backward at full size (256-row tiles,
    20 forward waves, staged dZ stores, grouped grad_hidden / grad_w tiles)
    give identical bits: every reduction has a fixed order and no persistent
    kernel races at this scale."""
    spec = workloads.spec_for(5)
    wl = workloads.build(spec, "cuda")
    h, w, y = wl.hidden, wl.w_vocab, wl.targets
    keep_seq = torch.ones(wl.B, dtype=torch.uint8)
    keep_seq[1::4] = 0
    row_keep = torch.repeat_interleave(keep_seq, torch.tensor(wl.seq_lens, dtype=torch.int64)).cuda()
    runs = []
    for _ in range(2):
        fw = mc.token_logprobs(h, w, y)
        bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], wl.advantages, None, row_keep=row_keep)
        torch.cuda.synchronize()
        runs.append((fw, bw))
    (fa, ba), (fb, bb) = runs
    for k in ("logp", "entropy", "lse"):
        assert torch.equal(fa[k], fb[k]), k
    assert torch.equal(ba["grad_hidden"], bb["grad_hidden"])
    assert torch.equal(ba["grad_w"], bb["grad_w"])
