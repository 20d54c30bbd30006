"""GPU sequence ratio statistics / MirrorPop mask (mc_seq_ratio_filter) vs the
fp64 oracle on the same fp32 log-prob arrays (filter-only parity), plus the
forward -> filter composition on the tiny config."""

import math

import numpy as np
import pytest
import torch

import oracle
from gpu_util import (MASK_BAND, TOL_LOGP, TOL_RATIO, assert_close_abs, assert_close_rel, assert_masks_match,
                      np_)
from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def compare(lp, lb, mask, cu, delta, delta_v):
    out = mc.seq_ratio_filter(lp.cuda(), lb.cuda(), None if mask is None else mask.cuda(), cu.cuda(), delta,
                              delta_v)
    torch.cuda.synchronize()
    ref = oracle.seq_ratio_filter(lp.numpy(), lb.numpy(), None if mask is None else mask.numpy(), cu.numpy(),
                                  float(np.float32(delta)), float(np.float32(delta_v)))
    np.testing.assert_array_equal(np_(out["n_tokens"]), ref["n_tokens"])
    # ratio-space statistics e^S (Eq. 18) and e^A (Eq. 20), relative error
    assert_close_rel(np.exp(np_(out["signed_mean"])), np.exp(ref["signed_mean"]), TOL_RATIO, "geo-mean ratio")
    assert_close_rel(np.exp(np_(out["abs_mean"])), np.exp(ref["abs_mean"]), TOL_RATIO, "MirrorPop ratio")
    assert_close_rel(np_(out["token_ratio"]), ref["token_ratio"], TOL_RATIO, "token ratio")
    assert_masks_match(np_(out["keep"]), ref["keep"], ref["abs_mean"], delta, MASK_BAND, "keep")
    if delta_v >= 0:
        assert_masks_match(np_(out["keep_vanilla"]), ref["keep_vanilla"], np.abs(ref["signed_mean"]), delta_v,
                           MASK_BAND, "keep_vanilla")
    else:
        assert not np_(out["keep_vanilla"]).any()
    # token_keep follows keep exactly (same decision reused), masked by loss_mask
    keep = np_(out["keep"]).astype(bool)
    cu_ = cu.numpy()
    seq = np.repeat(np.arange(len(cu_) - 1), np.diff(cu_))
    m = np.ones(lp.shape[0], dtype=bool) if mask is None else mask.numpy().astype(bool)
    np.testing.assert_array_equal(np_(out["token_keep"]).astype(bool), keep[seq] & m)
    return out, ref


def make(lens, gap_std=0.2, seed=0, mask_p=None, cancel=False):
    g = torch.Generator().manual_seed(seed)
    cu = torch.zeros(len(lens) + 1, dtype=torch.int64)
    cu[1:] = torch.cumsum(torch.tensor(lens, dtype=torch.int64), 0)
    N = int(cu[-1])
    lp = -torch.rand(N, generator=g) * 8.0
    per_seq = torch.randn(len(lens), generator=g) * gap_std
    gap = torch.repeat_interleave(per_seq, torch.tensor(lens)) + torch.randn(N, generator=g) * 0.05
    if cancel:
        sign = torch.tensor([1.0 if (k // 3) % 2 == 0 else -1.0 for k in range(N)])
        gap = 0.3 * sign
    lb = (lp.double() - gap.double()).float()
    mask = None if mask_p is None else (torch.rand(N, generator=g) < mask_p).to(torch.uint8)
    return lp.float(), lb, mask, cu


@pytest.mark.parametrize("delta,delta_v", [(0.0, -1.0), (0.02, 0.02), (0.05, 0.05), (0.1, 0.1), (0.2, 0.2),
                                           (math.log(2), 0.1)])
def test_config_shaped_sequences(delta, delta_v):
    lens = torch.randint(512, 8193, (32,), generator=torch.Generator().manual_seed(3)).tolist()
    compare(*make(lens, seed=1), delta, delta_v)


@pytest.mark.parametrize("mask_p", [None, 0.8])
def test_staged_chunks_odd_offsets_and_array_tail(mask_p):
    """Sequences staged in 4096-token chunks: one starting at an odd offset
    and spanning three chunks, an empty one, one of a single token, and an
    array length (12,295) that is not a multiple of 16, so the last tokens
    are past the last full 16 bytes; repeated calls agree bit for bit."""
    lens = [5, 0, 1, 8995, 3294]
    lp, lb, mask, cu = make(lens, seed=21, mask_p=mask_p)
    a, _ = compare(lp, lb, mask, cu, 0.1, 0.1)
    b = mc.seq_ratio_filter(lp.cuda(), lb.cuda(), None if mask is None else mask.cuda(), cu.cuda(), 0.1, 0.1)
    for k in a:
        assert torch.equal(a[k], b[k]), k


def test_masks_odd_offsets_empty_and_length_one():
    lens = [1, 0, 3, 5, 7, 0, 1, 130, 1023, 4, 9]  # odd starts exercise the scalar head/tail
    compare(*make(lens, seed=2, mask_p=0.6), 0.1, 0.1)


def test_all_tokens_masked_sequence():
    lp, lb, _, cu = make([10, 20, 30], seed=4)
    mask = torch.ones(60, dtype=torch.uint8)
    mask[10:30] = 0
    out, ref = compare(lp, lb, mask, cu, 0.3, 0.3)
    assert int(out["n_tokens"][1]) == 0 and int(out["keep"][1]) == 0


def test_cancellation_variant():
    """Alternating-sign gaps: Vanilla keeps, MirrorPop drops (the paper's case)."""
    lp, lb, mask, cu = make([64, 96, 120], cancel=True)
    out, ref = compare(lp, lb, mask, cu, 0.2, 0.2)
    assert np_(out["keep"]).sum() == 0 and np_(out["keep_vanilla"]).sum() >= 1


def test_identical_policies():
    lp, _, _, cu = make([100, 200, 3])
    out, _ = compare(lp, lp.clone(), None, cu, 0.0, 0.0)
    assert np_(out["keep"]).all() and np.all(np_(out["token_ratio"]) == 1.0)


def test_unaligned_pointers_take_the_scalar_path():
    lp, lb, mask, cu = make([33, 65, 2], seed=5, mask_p=0.5)
    big_lp = torch.zeros(lp.numel() + 1)
    big_lb = torch.zeros(lb.numel() + 1)
    big_lp[1:] = lp
    big_lb[1:] = lb
    d_lp, d_lb = big_lp.cuda()[1:], big_lb.cuda()[1:]  # 4-byte but not 16-byte aligned
    out = mc.seq_ratio_filter(d_lp, d_lb, mask.cuda(), cu.cuda(), 0.2, 0.2)
    ref = oracle.seq_ratio_filter(lp.numpy(), lb.numpy(), mask.numpy(), cu.numpy(), 0.2, 0.2)
    assert_close_rel(np.exp(np_(out["abs_mean"])), np.exp(ref["abs_mean"]), TOL_RATIO, "abs mean")


def test_forward_then_filter_tiny_config():
    """Tiny config end to end: behaviour = oracle policy log-probs + N(0, 0.05^2)."""
    wl = workloads.build(workloads.spec_for(1), "cpu")
    ref_lp = oracle.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)["logp"]
    lb = torch.from_numpy(ref_lp + wl.gap.double().numpy()).float()
    fw = mc.token_logprobs(wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda())
    delta = wl.spec.delta
    out = mc.seq_ratio_filter(fw["logp"], lb.cuda(), wl.loss_mask.cuda(), wl.cu_seqlens.cuda(), delta, delta)
    ref = oracle.seq_ratio_filter(ref_lp, lb.numpy(), wl.loss_mask.numpy(), wl.cu_seqlens.numpy(), delta, delta)
    # End to end the log-probs themselves differ by up to TOL_LOGP, so the band
    # around the threshold widens by each sequence's mean |dlogp|.
    dlogp = np.abs(np_(fw["logp"]) - ref_lp)
    assert dlogp.max() <= TOL_LOGP
    cu = wl.cu_seqlens.numpy()
    band = MASK_BAND + np.array([dlogp[cu[i]:cu[i + 1]].mean() for i in range(wl.B)])
    got, want = np_(out["keep"]).astype(bool), ref["keep"].astype(bool)
    assert not np.any((got != want) & (np.abs(ref["abs_mean"] - delta) > band))
    # delta = 0.04 (reading c1) sits inside the tiny config's spread of A_i: the
    # filter both keeps and drops sequences.
    assert 0 < want.sum() < wl.B, want


def test_many_tiny_sequences():
    """100,003 sequences of 0-5 tokens (most shorter than one 16-byte vector,
    many empty): every persistent CTA strides over dozens of sequences, and
    the head / vector / tail split of each sequence is exercised at every
    offset."""
    lens = torch.randint(0, 6, (100_003,), generator=torch.Generator().manual_seed(11)).tolist()
    compare(*make(lens, seed=12, mask_p=0.8), 0.1, 0.1)
