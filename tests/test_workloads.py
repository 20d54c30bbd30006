"""The seeded generator: shapes, determinism and the stated distributions."""

import math

import torch

from paper_2606_04847_gb300 import workloads


def test_config1_shapes_and_determinism():
    a = workloads.build(workloads.spec_for(1), "cpu")
    b = workloads.build(workloads.spec_for(1), "cpu")
    assert a.hidden.shape == (256, 512) and a.hidden.dtype == torch.bfloat16
    assert a.w_vocab.shape == (4096, 512) and a.w_vocab.dtype == torch.bfloat16
    assert a.targets.dtype == torch.int32 and a.cu_seqlens.tolist() == list(range(0, 257, 32))
    for k in ("hidden", "w_vocab", "targets", "gap", "loss_mask"):
        assert torch.equal(getattr(a, k), getattr(b, k)), k
    # W ~ N(0, 1/d): std 1/sqrt(512)
    assert abs(a.w_vocab.float().std().item() * math.sqrt(512) - 1) < 0.02
    assert abs(a.hidden.float().std().item() - 1) < 0.02
    assert abs(a.gap.std().item() - 0.05) < 0.01


def test_sampled_targets_follow_softmax_on_small_case():
    """Gumbel-max draws at a peaked small case land on the argmax most often."""
    spec = workloads.spec_for(2, n_seqs=2, len_lo=64, len_hi=64, d=64, V=97, w_scale=8.0)
    wl = workloads.build(spec, "cpu")
    z = wl.hidden.float() @ wl.w_vocab.float().T
    agree = (z.argmax(1).to(torch.int32) == wl.targets).float().mean().item()
    assert agree > 0.5
    assert int(wl.targets.min()) >= 0 and int(wl.targets.max()) < 97


def test_sequence_gap_and_subset_gap():
    spec = workloads.spec_for(3, n_seqs=6, len_lo=5, len_hi=9, d=16, V=32)
    wl = workloads.build(spec, "cpu")
    cu = wl.cu_seqlens.tolist()
    for i in range(6):
        seg = wl.gap[cu[i]:cu[i + 1]]
        assert torch.all(seg == seg[0])
    spec2 = workloads.spec_for(2, n_seqs=20, len_lo=4, len_hi=4, d=16, V=32)
    wl2 = workloads.build(spec2, "cpu")
    nz = sum(1 for i in range(20) if torch.any(wl2.gap[4 * i:4 * i + 4] != 0))
    assert nz == 2  # ceil(10 % of 20)


def test_multi_turn_mask_structure():
    spec = workloads.spec_for(4, n_seqs=5, len_lo=50, len_hi=80, d=16, V=32)
    wl = workloads.build(spec, "cpu")
    first = workloads.build(spec, "cpu", first_turn_only=True)
    assert torch.all(first.loss_mask <= wl.loss_mask)
    cu = wl.cu_seqlens.tolist()
    for i in range(5):
        m = wl.loss_mask[cu[i]:cu[i + 1]]
        assert m[0] == 0 and m[-1] == 1  # every turn opens with prompt and ends with response


def test_zero_length_sequences_and_cancellation_variant():
    spec = workloads.spec_for(3, d=16, V=32)
    wl = workloads.build(spec, "cpu", lengths=[3, 0, 8, 0])
    assert wl.N == 11 and wl.cu_seqlens.tolist() == [0, 3, 3, 11, 11]
    gap = workloads.cancellation_gap(wl, magnitude=0.3, frac=0.5, run=2)
    assert gap.shape == wl.gap.shape
