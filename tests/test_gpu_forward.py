"""GPU forward (mc_token_logprobs) vs the fp64 oracle, element by element.

Sizes span several 128-row blocks and 256-column vocabulary tiles, with
ragged tails in both, the tiny config at full size, and the edge cases:
N = 1, V not a multiple of the tile, V < one tile, targets at 0 and V-1,
peaked softmax (low entropy), temperature, d from 64 to 8192.
"""

import math

import numpy as np
import pytest
import torch

import oracle
from gpu_util import TOL_ENT, TOL_LOGP, assert_close_abs, np_
from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def run_and_compare(wl, inv_temp=1.0, targets=None):
    h = wl.hidden.cuda()
    w = wl.w_vocab.cuda()
    y = (wl.targets if targets is None else targets).cuda()
    out = mc.token_logprobs(h, w, y, inv_temp)
    torch.cuda.synchronize()
    ref = oracle.token_logprobs(wl.hidden, wl.w_vocab, y.cpu(), inv_temp)
    assert_close_abs(np_(out["logp"]), ref["logp"], TOL_LOGP, "logp")
    assert_close_abs(np_(out["entropy"]), ref["entropy"], TOL_ENT, "entropy")
    assert_close_abs(np_(out["lse"]), ref["lse"], TOL_LOGP, "lse")
    return out, ref


def test_config1_tiny_full_size():
    wl = workloads.build(workloads.spec_for(1), "cpu")
    run_and_compare(wl)


@pytest.mark.parametrize("N,d,V", [
    (1, 64, 300),            # single row, V < 2 tiles with a tail
    (300, 128, 4097),        # ragged rows (3 blocks) and one-column vocab tail
    (129, 256, 200),         # V smaller than one tile
    (520, 512, 151936 // 16),  # 9496 = 37 tiles + 24 columns
    (257, 5120, 1024),       # the 27B-class hidden size
    (130, 6144, 777),        # 96 k-blocks per tile
    (300, 8192, 1000),       # 128 k-blocks per tile
])
def test_ragged_shapes(N, d, V):
    spec = workloads.spec_for(1, n_seqs=1, len_lo=N, len_hi=N, d=d, V=V)
    run_and_compare(workloads.build(spec, "cpu"))


@pytest.mark.parametrize("inv_temp", [1.0, 1.0 / 0.9])
def test_wide_tiles_ragged(inv_temp):
    """>= 2304 rows: 256-row tiles with 16 epilogue warps over two column
    halves when twice the splits fit the workspace, else 8 (4500 rows = 17
    blocks + 148), a vocabulary tail of 184 columns."""
    spec = workloads.spec_for(1, n_seqs=1, len_lo=4500, len_hi=4500, d=256, V=3000)
    run_and_compare(workloads.build(spec, "cpu"), inv_temp=inv_temp)


def test_million_entry_vocabulary():
    """V = 1,000,003 (3,907 tiles, a 3-column tail; the maximum 16 splits per
    row block) on 64 rows, d = 64."""
    spec = workloads.spec_for(1, n_seqs=1, len_lo=64, len_hi=64, d=64, V=1_000_003, seed=26)
    run_and_compare(workloads.build(spec, "cpu"))


@pytest.mark.parametrize("N", [2048, 2304, 3000])
def test_wide_tile_threshold(N):
    """The row counts around the switch to 256-row tiles (at 2304 rows):
    2048 rows on 128-row tiles, exactly 9 wide row blocks, and 11 + 184."""
    spec = workloads.spec_for(1, n_seqs=1, len_lo=N, len_hi=N, d=256, V=2000, seed=28)
    run_and_compare(workloads.build(spec, "cpu"))


def test_wide_tiles_long_hidden():
    """256-row tiles with d = 8192 (128 k-blocks through the 3-stage ring per
    tile): 4200 rows = 16 blocks + 104, V = 300 (a 44-column tail)."""
    spec = workloads.spec_for(1, n_seqs=1, len_lo=4200, len_hi=4200, d=8192, V=300, seed=23)
    run_and_compare(workloads.build(spec, "cpu"))


def test_wide_tiles_tiny_vocabulary_single_k_block():
    """256-row tiles with V = 17 (less than one 32-column chunk) and d = 64
    (one k-block per tile)."""
    spec = workloads.spec_for(1, n_seqs=1, len_lo=4500, len_hi=4500, d=64, V=17)
    run_and_compare(workloads.build(spec, "cpu"))


@pytest.mark.parametrize("N,V", [(127, 1), (128, 31), (129, 33), (5, 257)])
def test_tiny_vocabularies_and_block_edges(N, V):
    """V = 1 (logp = 0, entropy = 0), V inside the first 32-column chunk, N on
    both sides of a 128-row block."""
    spec = workloads.spec_for(1, n_seqs=1, len_lo=N, len_hi=N, d=64, V=V)
    out, ref = run_and_compare(workloads.build(spec, "cpu"))
    if V == 1:
        # Exactly 0 in real arithmetic. The kernel works in base 2: it keeps
        # m = z log2(e) and returns lse = ln(2) (m + log2 s) with s = 1, so
        # z_y - lse is z (1 - ln(2) log2(e)) after two fp32 roundings, a few
        # ulps of |z| (|z| < 8 here): about 1e-6, bounded by 1e-5.
        assert np.abs(np_(out["logp"])).max() < 1e-5 and np.abs(np_(out["entropy"])).max() < 1e-5


def test_targets_at_vocab_edges_and_temperature():
    spec = workloads.spec_for(1, n_seqs=2, len_lo=150, len_hi=150, d=256, V=1000)
    wl = workloads.build(spec, "cpu")
    y = wl.targets.clone()
    y[::3] = 0
    y[1::3] = 999
    run_and_compare(wl, inv_temp=1.0 / 0.9, targets=y)


def test_peaked_softmax_low_entropy():
    """W scaled x8: logits std ~8, entropies spread over ~[0, 3] nats."""
    spec = workloads.spec_for(1, n_seqs=2, len_lo=200, len_hi=200, d=512, V=3000, w_scale=8.0)
    out, ref = run_and_compare(workloads.build(spec, "cpu"))
    assert ref["entropy"].min() < 0.5


@pytest.mark.parametrize("N", [300, 4500])  # 128-row and 256-row tiles
def test_extreme_logits(N):
    """W x 64: logits spread over hundreds of units, so nearly every row is
    one-hot-dominant and the running maximum jumps between tiles; exp2 of
    very negative arguments flushes to 0."""
    spec = workloads.spec_for(1, n_seqs=1, len_lo=N, len_hi=N, d=128, V=2000, w_scale=64.0)
    out, ref = run_and_compare(workloads.build(spec, "cpu"))
    assert ref["entropy"].min() < 1e-3


def test_uniform_logits():
    """W = 0: every logit equal; logp = -log V and entropy = log V."""
    N, d, V = 130, 64, 777
    h = torch.randn(N, d).to(torch.bfloat16).cuda()
    w = torch.zeros(V, d, dtype=torch.bfloat16).cuda()
    y = torch.randint(0, V, (N,), dtype=torch.int32).cuda()
    out = mc.token_logprobs(h, w, y)
    assert_close_abs(np_(out["logp"]), np.full(N, -math.log(V)), 1e-5, "logp")
    assert_close_abs(np_(out["entropy"]), np.full(N, math.log(V)), 1e-4, "entropy")


def test_out_of_range_target_sets_status_and_nan():
    spec = workloads.spec_for(1, n_seqs=1, len_lo=40, len_hi=40, d=64, V=500)
    wl = workloads.build(spec, "cpu")
    y = wl.targets.clone()
    y[3] = 500
    y[7] = -1
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = mc.token_logprobs(wl.hidden.cuda(), wl.w_vocab.cuda(), y.cuda(), dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & mc.MC_DEV_TARGET_RANGE
    lp = np_(out["logp"])
    assert np.isnan(lp[3]) and np.isnan(lp[7])
    good = np.ones(40, dtype=bool)
    good[[3, 7]] = False
    ref = oracle.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    assert_close_abs(lp[good], ref["logp"][good], TOL_LOGP, "logp of valid rows")


def test_deterministic_bitwise():
    wl = workloads.build(workloads.spec_for(1, n_seqs=3, len_lo=100, len_hi=100, d=512, V=5000), "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    a = mc.token_logprobs(h, w, y)
    b = mc.token_logprobs(h, w, y)
    for k in a:
        assert torch.equal(a[k], b[k]), k


def test_nullable_outputs_and_zero_rows():
    wl = workloads.build(workloads.spec_for(1, n_seqs=1, len_lo=64, len_hi=64, d=64, V=256), "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    full = mc.token_logprobs(h, w, y)
    only = mc.token_logprobs(h, w, y, out={"logp": torch.empty(64, device="cuda")})
    assert torch.equal(full["logp"], only["logp"])
    empty = mc.token_logprobs(h[:0], w, y[:0])
    assert empty["logp"].numel() == 0


def test_bounded_wait_selftest_keeps_context_usable():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    mc.selftest_bounded_wait(st, 20_000_000)  # 20 ms
    torch.cuda.synchronize()
    assert int(st.item()) & mc.MC_DEV_TIMEOUT
    test_config1_tiny_full_size()  # the context is still healthy


def test_binding_rejects_mis_shaped_outputs_and_workspaces():
    """Caller-supplied outputs and workspaces are checked before any launch: a
    wrong shape, dtype or layout raises instead of letting a kernel write past
    a buffer."""
    wl = workloads.build(workloads.spec_for(1, n_seqs=1, len_lo=64, len_hi=64, d=64, V=256), "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    with pytest.raises(ValueError):
        mc.token_logprobs(h, w, y, out={"logp": torch.empty(63, device="cuda")})
    with pytest.raises(TypeError):
        mc.token_logprobs(h, w, y, out={"logp": torch.empty(64, device="cuda", dtype=torch.float64)})
    with pytest.raises(TypeError):
        mc.token_logprobs(h, w, y, workspace=torch.empty(1 << 20, device="cuda", dtype=torch.float32))
    with pytest.raises(ValueError):
        mc.token_logprobs(h, w.t().contiguous().t(), y)  # a strided view of W
    fw = mc.token_logprobs(h, w, y)
    g = torch.randn(64, device="cuda")
    with pytest.raises(ValueError):
        mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g, grad_w=torch.empty(256, 32, device="cuda"))
    with pytest.raises(ValueError):
        mc.token_logprobs_bwd(h, w, y, fw["lse"][:10], fw["entropy"], g)
    cu = torch.tensor([0, 64], dtype=torch.int64, device="cuda")
    with pytest.raises(ValueError):
        mc.seq_ratio_filter(fw["logp"], fw["logp"][:32], None, cu, 0.1)
