"""Parity at the configured full sizes, in the launch configuration bench.py
times (whole batches through the C ABI, default workspaces).

* forward: every row runs on the GPU; at least 256 rows per configuration are
  recomputed by the fp64 oracle, chosen to cover every (128-row sub-block,
  TMEM lane quadrant) position of a 256-row tile, the ragged last row block,
  and targets in both column halves of a vocabulary tile.
* filter: the full batch of sequences, filter-only parity (both sides get the
  same fp32 log-prob arrays with the config's lengths, gaps and masks).
* backward at the 9B-class shape (d = 4096, V = 248,320): 4,500 live rows
  picked by row_keep from the full workload (256-row tiles everywhere, grad_w's
  970 x 16 output tiles with its tile grouping, a ragged last K block), every
  grad_hidden row and 512 grad_w vocabulary rows compared element by element
  with the oracle.
* the chain bench.py times (forward -> filter token_keep -> backward row_keep)
  on the whole 9B-class batch: the oracle recomputes two whole sequences (one
  kept, one dropped by Eq. 21) from their hidden states, their MirrorPop
  statistics and keep decisions, and 256 of their grad_hidden rows; grad_w,
  which sums over all ~90k kept rows, is checked through identities that hold
  at any size: <grad_hidden, H> = <grad_w, W> and sum_v grad_w[v, :] = 0.
* the 27B-class batch end to end through the filter with its per-turn loss
  mask, and the mid and 9B-class forward workloads end to end through the
  filter: the oracle recomputes a kept and a dropped sequence whole.
"""

import numpy as np
import pytest
import torch

import oracle
from gpu_util import (MASK_BAND, TOL_ENT, TOL_GRAD, TOL_LOGP, TOL_RATIO, assert_close_abs, assert_close_rel,
                      assert_masks_match, np_, rel_fro)
from paper_2606_04847_gb300 import mc, workloads

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

TILE_ROWS = 256   # rows of a wide tile: two 128-row sub-blocks x four 32-lane quadrants
TILE_COLS = 256   # vocabulary columns of a tile: two column halves of 128


def coverage_rows(n, targets, k=256, seed=0):
    """At least k rows: 24 per (sub-block, lane quadrant) position of a
    256-row tile (8 positions), 16 from the last (partial) row block, plus
    rows whose target lies in each column half of a vocabulary tile."""
    g = np.random.default_rng(seed)
    pos = (np.arange(n) % TILE_ROWS) // 32
    rows = set([0, n - 1])
    for p in range(8):
        cand = np.nonzero(pos == p)[0]
        rows.update(g.choice(cand, size=min(24, len(cand)), replace=False).tolist())
    last = np.arange((n - 1) // TILE_ROWS * TILE_ROWS, n)
    rows.update(g.choice(last, size=min(16, len(last)), replace=False).tolist())
    half = (targets % TILE_COLS) >= TILE_COLS // 2
    for h in (False, True):
        cand = np.nonzero(half == h)[0]
        rows.update(g.choice(cand, size=min(16, len(cand)), replace=False).tolist())
    rest = np.setdiff1d(np.arange(n), np.fromiter(rows, dtype=np.int64))
    if len(rows) < k:
        rows.update(g.choice(rest, size=min(k - len(rows), len(rest)), replace=False).tolist())
    return np.array(sorted(rows))


@pytest.mark.parametrize("config", [2, 3, 4, 5])
def test_forward_full_size(config):
    spec = workloads.spec_for(config)
    wl = workloads.build(spec, "cuda")
    out = mc.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    torch.cuda.synchronize()
    y_all = np_(wl.targets).astype(np.int64)
    rows = coverage_rows(wl.N, y_all, seed=config)
    assert len(rows) >= 256
    assert set(((rows % TILE_ROWS) // 32).tolist()) == set(range(8))
    assert rows.max() == wl.N - 1 and (rows >= (wl.N - 1) // TILE_ROWS * TILE_ROWS).sum() >= 2
    assert {bool(v) for v in (y_all[rows] % TILE_COLS) >= TILE_COLS // 2} == {False, True}
    ridx = torch.from_numpy(rows).cuda()
    w64 = wl.w_vocab.cpu().double().numpy()  # exact upcast, once
    ref = oracle.token_logprobs(wl.hidden[ridx].cpu(), w64, wl.targets[ridx].cpu(), spec.inv_temperature,
                                rows_per_block=TILE_ROWS)
    del w64
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


def test_backward_full_shape_elementwise():
    """9B-class shape, 4,500 live rows (17 row blocks of 256 + 148) picked by
    row_keep from the full workload: every grad_hidden row and 512 grad_w
    vocabulary rows against the oracle at the stated 1e-2 relative bound."""
    spec = workloads.spec_for(5)
    wl = workloads.build(spec, "cuda")
    h, w, y = wl.hidden, wl.w_vocab, wl.targets
    g = np.random.default_rng(55)
    live = np.sort(g.choice(wl.N, size=4500, replace=False))
    live[-1] = wl.N - 1
    live = np.unique(live)
    row_keep = torch.zeros(wl.N, dtype=torch.uint8)
    row_keep[torch.from_numpy(live)] = 1
    fw = mc.token_logprobs(h, w, y)
    bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], wl.advantages, None, row_keep=row_keep.cuda())
    torch.cuda.synchronize()
    gh, gw = bw["grad_hidden"], bw["grad_w"]
    assert torch.isfinite(gw).all()

    # Vocabulary rows: 128 targets of live rows, the first and last rows, and
    # random rows; every (sub-block, lane quadrant) position of grad_w's
    # 256-row tiles appears.
    y_live = np_(y[torch.from_numpy(live).cuda()]).astype(np.int64)
    vrows = set(g.choice(np.unique(y_live), size=128, replace=False).tolist())
    vrows.update([0, spec.V - 1, 255, 256])
    vrows.update(g.choice(spec.V, size=512 - len(vrows), replace=False).tolist())
    vrows = np.array(sorted(vrows))
    assert len(vrows) >= 500 and set(((vrows % TILE_ROWS) // 32).tolist()) == set(range(8))

    lidx = torch.from_numpy(live).cuda()
    w64 = w.cpu().double().numpy()
    ref = oracle.token_logprobs_bwd_rows(h[lidx].cpu(), w64, y[lidx].cpu(), wl.advantages[lidx].cpu(),
                                         vocab_rows=vrows)
    del w64
    got_h = np_(gh[lidx].float())
    for i, r in enumerate(live):
        e = rel_fro(got_h[i], ref["grad_hidden"][i])
        assert e <= TOL_GRAD, f"grad_hidden row {r}: rel err {e:.3e}"
    assert rel_fro(got_h, ref["grad_hidden"]) <= TOL_GRAD
    dropped = torch.ones(wl.N, dtype=torch.bool)
    dropped[torch.from_numpy(live)] = False
    assert torch.count_nonzero(gh[dropped.cuda()]) == 0
    got_w = np_(gw[torch.from_numpy(vrows).cuda()])
    for i, v in enumerate(vrows):
        e = rel_fro(got_w[i], ref["grad_w"][i])
        assert e <= TOL_GRAD, f"grad_w row {v}: rel err {e:.3e}"
    assert rel_fro(got_w, ref["grad_w"]) <= TOL_GRAD


def test_chain_full_size_9b():
    """The step bench.py times, on the whole 9B-class batch: forward ->
    MirrorPop filter (behaviour = policy + the per-sequence gap) -> backward
    with the filter's token_keep as row_keep. The oracle recomputes the
    shortest kept and the shortest dropped sequence from their hidden
    states."""
    spec = workloads.spec_for(5)
    wl = workloads.build(spec, "cuda")
    h, w, y = wl.hidden, wl.w_vocab, wl.targets
    fw = mc.token_logprobs(h, w, y)
    lb = fw["logp"] + wl.gap
    flt = mc.seq_ratio_filter(fw["logp"], lb, wl.loss_mask, wl.cu_seqlens, spec.delta, spec.delta)
    bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], wl.advantages, None, row_keep=flt["token_keep"])
    torch.cuda.synchronize()
    gh, gw = bw["grad_hidden"], bw["grad_w"]
    assert torch.isfinite(gw).all()

    # Two whole sequences through the oracle: with logp_behaviour = logp_policy
    # + gap_i, A_i = |gap_i| (Eq. 20), so |gap_i| far from delta picks one
    # sequence each side of Eq. 21's threshold.
    cu = np_(wl.cu_seqlens)
    gap = np_(wl.gap)[cu[:-1]]
    lens = np.diff(cu)
    far = np.abs(np.abs(gap) - spec.delta) > 0.02
    kept_i = min(np.nonzero(far & (np.abs(gap) < spec.delta))[0], key=lambda i: lens[i])
    drop_i = min(np.nonzero(far & (np.abs(gap) > spec.delta))[0], key=lambda i: lens[i])
    seqs = [kept_i, drop_i]
    rows = np.concatenate([np.arange(cu[i], cu[i + 1]) for i in seqs])
    ridx = torch.from_numpy(rows).cuda()
    w64 = w.cpu().double().numpy()
    h_rows, y_rows = h[ridx].cpu(), y[ridx].cpu()
    ref_f = oracle.token_logprobs(h_rows, w64, y_rows, rows_per_block=TILE_ROWS)
    assert_close_abs(np_(fw["logp"][ridx]), ref_f["logp"], TOL_LOGP, "chain logp")
    sub_cu = np.concatenate([[0], np.cumsum(lens[seqs])])
    gap_rows = np_(wl.gap[ridx]).astype(np.float64)
    mask_rows = np_(wl.loss_mask[ridx])
    ref_flt = oracle.seq_ratio_filter(ref_f["logp"], ref_f["logp"] + gap_rows, mask_rows, sub_cu,
                                      float(np.float32(spec.delta)))
    assert list(ref_flt["keep"]) == [1, 0]
    got_keep = np_(flt["keep"])[seqs]
    dlogp = np.abs(np_(fw["logp"][ridx]) - ref_f["logp"])
    band = MASK_BAND + np.array([dlogp[sub_cu[k]:sub_cu[k + 1]].mean() for k in range(2)])
    assert_masks_match(got_keep, ref_flt["keep"], ref_flt["abs_mean"], spec.delta, band, "chain keep")
    assert_close_rel(np.exp(np_(flt["abs_mean"])[seqs]), np.exp(ref_flt["abs_mean"]), TOL_RATIO, "chain e^A")

    # 256 grad_hidden rows: 192 of the kept sequence, 64 of the dropped one
    # (which must be exactly zero). The oracle's upstream gradient is the
    # advantage weight gated by its own token_keep.
    g = np.random.default_rng(56)
    n_k = lens[kept_i]
    pick = np.sort(np.concatenate([g.choice(n_k, size=192, replace=False),
                                   n_k + g.choice(lens[drop_i], size=64, replace=False)]))
    g_rows = np_(wl.advantages[ridx]).astype(np.float64)[pick] * ref_flt["token_keep"][pick]
    tpick = torch.from_numpy(pick)
    ref_b = oracle.token_logprobs_bwd_rows(h_rows[tpick], w64, y_rows[tpick], g_rows, vocab_rows=[])
    del w64
    got = np_(gh[ridx[tpick.cuda()]].float())
    for i, r in enumerate(rows[pick]):
        if g_rows[i] == 0:
            assert not got[i].any(), f"dropped row {r} has a gradient"
        else:
            e = rel_fro(got[i], ref_b["grad_hidden"][i])
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


def test_chain_27b_whole_sequences():
    """27B-class batch (d = 5120, multi-turn sequences, the prompt tokens of
    every turn masked out of the loss): forward over all 595k tokens, then the
    MirrorPop filter with the per-turn loss mask. The oracle recomputes the
    shortest kept and the shortest dropped sequence whole from their hidden
    states: every log-prob, the masked token count L_i, the Eq. 20 statistic
    and the Eq. 21 decision."""
    spec = workloads.spec_for(4)
    wl = workloads.build(spec, "cuda")
    fw = mc.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    lb = fw["logp"] + wl.gap
    flt = mc.seq_ratio_filter(fw["logp"], lb, wl.loss_mask, wl.cu_seqlens, spec.delta, spec.delta)
    torch.cuda.synchronize()
    cu = np_(wl.cu_seqlens)
    gap = np_(wl.gap)[cu[:-1]]
    lens = np.diff(cu)
    far = np.abs(np.abs(gap) - spec.delta) > 0.02
    kept_i = min(np.nonzero(far & (np.abs(gap) < spec.delta))[0], key=lambda i: lens[i])
    drop_i = min(np.nonzero(far & (np.abs(gap) > spec.delta))[0], key=lambda i: lens[i])
    seqs = [kept_i, drop_i]
    rows = np.concatenate([np.arange(cu[i], cu[i + 1]) for i in seqs])
    ridx = torch.from_numpy(rows).cuda()
    w64 = wl.w_vocab.cpu().double().numpy()
    ref_f = oracle.token_logprobs(wl.hidden[ridx].cpu(), w64, wl.targets[ridx].cpu(), rows_per_block=TILE_ROWS)
    del w64
    assert_close_abs(np_(fw["logp"][ridx]), ref_f["logp"], TOL_LOGP, "27B logp")
    assert_close_abs(np_(fw["entropy"][ridx]), ref_f["entropy"], TOL_ENT, "27B entropy")
    sub_cu = np.concatenate([[0], np.cumsum(lens[seqs])])
    mask_rows = np_(wl.loss_mask[ridx])
    ref_flt = oracle.seq_ratio_filter(ref_f["logp"], ref_f["logp"] + np_(wl.gap[ridx]).astype(np.float64),
                                      mask_rows, sub_cu, float(np.float32(spec.delta)))
    assert list(ref_flt["keep"]) == [1, 0]
    assert 0 < ref_flt["n_tokens"][0] < lens[kept_i]  # the prompt tokens of every turn are masked out
    np.testing.assert_array_equal(np_(flt["n_tokens"])[seqs], ref_flt["n_tokens"])
    dlogp = np.abs(np_(fw["logp"][ridx]) - ref_f["logp"])
    band = MASK_BAND + np.array([dlogp[sub_cu[k]:sub_cu[k + 1]].mean() for k in range(2)])
    assert_masks_match(np_(flt["keep"])[seqs], ref_flt["keep"], ref_flt["abs_mean"], spec.delta, band, "27B keep")
    assert_close_rel(np.exp(np_(flt["abs_mean"])[seqs]), np.exp(ref_flt["abs_mean"]), TOL_RATIO, "27B e^A")
    tk = np_(flt["token_keep"][ridx]).astype(bool)
    np.testing.assert_array_equal(tk, ref_flt["token_keep"].astype(bool))


@pytest.mark.parametrize("config", [2, 3])
def test_chain_forward_workloads_whole_sequences(config):
    """The mid (per-token behaviour gap on 10 % of sequences) and 9B-class
    forward workloads end to end: forward over the whole batch, then the
    filter; the oracle recomputes one kept and one dropped sequence whole
    (chosen from the synthetic gap: with logp_behaviour = logp_policy + gap,
    A_i is the mean |gap| over the sequence's loss-masked tokens)."""
    spec = workloads.spec_for(config)
    wl = workloads.build(spec, "cuda")
    fw = mc.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    lb = fw["logp"] + wl.gap
    flt = mc.seq_ratio_filter(fw["logp"], lb, wl.loss_mask, wl.cu_seqlens, spec.delta, spec.delta)
    torch.cuda.synchronize()
    cu = np_(wl.cu_seqlens)
    lens = np.diff(cu)
    gap, m = np.abs(np_(wl.gap).astype(np.float64)), np_(wl.loss_mask).astype(bool)
    a_gap = np.array([gap[cu[i]:cu[i + 1]][m[cu[i]:cu[i + 1]]].mean() for i in range(wl.B)])
    far = np.abs(a_gap - spec.delta) > 0.01
    kept_i = min(np.nonzero(far & (a_gap < spec.delta))[0], key=lambda i: lens[i])
    drop_i = min(np.nonzero(far & (a_gap > spec.delta))[0], key=lambda i: lens[i])
    seqs = [kept_i, drop_i]
    rows = np.concatenate([np.arange(cu[i], cu[i + 1]) for i in seqs])
    ridx = torch.from_numpy(rows).cuda()
    w64 = wl.w_vocab.cpu().double().numpy()
    ref_f = oracle.token_logprobs(wl.hidden[ridx].cpu(), w64, wl.targets[ridx].cpu(), rows_per_block=TILE_ROWS)
    del w64
    assert_close_abs(np_(fw["logp"][ridx]), ref_f["logp"], TOL_LOGP, f"config {config} logp")
    assert_close_abs(np_(fw["entropy"][ridx]), ref_f["entropy"], TOL_ENT, f"config {config} entropy")
    sub_cu = np.concatenate([[0], np.cumsum(lens[seqs])])
    ref_flt = oracle.seq_ratio_filter(ref_f["logp"], ref_f["logp"] + np_(wl.gap[ridx]).astype(np.float64),
                                      np_(wl.loss_mask[ridx]), sub_cu, float(np.float32(spec.delta)),
                                      float(np.float32(spec.delta)))
    assert list(ref_flt["keep"]) == [1, 0]
    if config == 2:
        # A per-token gap of mean ~0: the signed statistic cancels (Vanilla
        # keeps the sequence) while the absolute one does not (MirrorPop drops it).
        assert ref_flt["keep_vanilla"][1] == 1
    np.testing.assert_array_equal(np_(flt["n_tokens"])[seqs], ref_flt["n_tokens"])
    dlogp = np.abs(np_(fw["logp"][ridx]) - ref_f["logp"])
    band = MASK_BAND + np.array([dlogp[sub_cu[k]:sub_cu[k + 1]].mean() for k in range(2)])
    assert_masks_match(np_(flt["keep"])[seqs], ref_flt["keep"], ref_flt["abs_mean"], spec.delta, band, "keep")
    assert_masks_match(np_(flt["keep_vanilla"])[seqs], ref_flt["keep_vanilla"], np.abs(ref_flt["signed_mean"]),
                       spec.delta, band, "keep_vanilla")
    assert_close_rel(np.exp(np_(flt["abs_mean"])[seqs]), np.exp(ref_flt["abs_mean"]), TOL_RATIO, "e^A")
    assert_close_rel(np.exp(np_(flt["signed_mean"])[seqs]), np.exp(ref_flt["signed_mean"]), TOL_RATIO, "e^S")


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
