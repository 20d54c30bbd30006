"""GPU backward (mc_token_logprobs_bwd) vs the fp64 oracle's closed form.

Relative Frobenius error of grad_hidden and grad_w <= 1e-2, and the same
bound on every grad_hidden row with a nonzero upstream gradient, over ragged shapes, several
row chunks (small workspace), accumulation into grad_w, the entropy term,
temperature and rows skipped by the keep-mask (zero upstream gradient).
"""

import numpy as np
import pytest
import torch

import oracle
from gpu_util import TOL_GRAD, np_, rel_fro
from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def setup(N, d, V, seed=0, w_scale=1.0):
    spec = workloads.spec_for(1, n_seqs=1, len_lo=N, len_hi=N, d=d, V=V, seed=seed, w_scale=w_scale)
    wl = workloads.build(spec, "cpu")
    g = torch.Generator().manual_seed(seed + 100)
    grad_logp = torch.randn(N, generator=g)
    grad_ent = torch.randn(N, generator=g) * 0.3
    return wl, grad_logp, grad_ent


def check(wl, grad_logp, grad_ent, inv_temp=1.0, rows_per_chunk=None, accumulate_base=None):
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    fw = mc.token_logprobs(h, w, y, inv_temp)
    gw = None
    if accumulate_base is not None:
        gw = accumulate_base.clone().cuda()
    out = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], grad_logp.cuda(),
                                None if grad_ent is None else grad_ent.cuda(), inv_temp,
                                rows_per_chunk=rows_per_chunk, grad_w=gw, accumulate=accumulate_base is not None)
    torch.cuda.synchronize()
    ref = oracle.token_logprobs_bwd(wl.hidden, wl.w_vocab, wl.targets, grad_logp,
                                    None if grad_ent is None else grad_ent, inv_temp)
    gh = np_(out["grad_hidden"].float())
    gwv = np_(out["grad_w"])
    want_w = ref["grad_w"] + (0 if accumulate_base is None else accumulate_base.double().numpy())
    e_h = rel_fro(gh, ref["grad_hidden"])
    e_w = rel_fro(gwv, want_w)
    assert e_h <= TOL_GRAD, f"grad_hidden rel err {e_h:.3e}"
    assert e_w <= TOL_GRAD, f"grad_w rel err {e_w:.3e}"
    nzmask = (grad_logp != 0).numpy()
    if grad_ent is not None:
        nzmask |= (grad_ent != 0).numpy()
    # Every row with a nonzero upstream gradient, at the stated bound.
    for r in np.nonzero(nzmask)[0]:
        er = rel_fro(gh[r], ref["grad_hidden"][r])
        assert er <= TOL_GRAD, f"row {r}: rel err {er:.3e}"
    return out, ref


def test_small_ragged():
    check(*setup(300, 128, 1000))


def test_tiny_config_shape_with_entropy_and_temperature():
    check(*setup(256, 512, 4096, seed=1), inv_temp=1.0 / 0.9)


def test_logp_only_upstream():
    wl, g, _ = setup(200, 256, 3000, seed=2)
    check(wl, g, None)


def test_multiple_row_chunks_and_accumulate():
    wl, g, ge = setup(450, 128, 700, seed=3)
    base = torch.randn(700, 128, generator=torch.Generator().manual_seed(9))
    check(wl, g, ge, rows_per_chunk=128, accumulate_base=base)


def test_rows_dropped_by_keep_mask_have_zero_gradient():
    wl, g, _ = setup(384, 128, 2000, seed=4)
    g[128:256] = 0.0  # a dropped sequence
    out, ref = check(wl, g, None)
    assert torch.count_nonzero(out["grad_hidden"][128:256]) == 0


def test_vocab_tail_and_large_hidden():
    check(*setup(130, 5120, 300, seed=5))


def test_single_entry_vocabulary_has_zero_gradient():
    wl, g, ge = setup(129, 64, 1, seed=8)
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    fw = mc.token_logprobs(h, w, y)
    out = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g.cuda(), ge.cuda())
    torch.cuda.synchronize()
    # p = 1 up to the rounding of exp2(z - lse): the gradient vanishes to ~1e-17
    assert out["grad_hidden"].float().abs().max() < 1e-6 and out["grad_w"].abs().max() < 1e-6


def test_million_entry_vocabulary():
    """V = 1,000,003: dZ rows of 2 MB, grad_hidden's K loop over 15,625
    k-blocks (256-row tiles), 3,907 grad_w row tiles; 64 rows, d = 64."""
    check(*setup(64, 64, 1_000_003, seed=27))


def test_long_hidden_8192():
    """d = 8192: 128 k-blocks per dZ tile and a 32-tile grad_hidden output
    row (128-row tiles: 300 rows), V = 600."""
    check(*setup(300, 8192, 600, seed=24))


def test_wide_tile_dz_long_hidden():
    """256-row dZ tiles at d = 8192 (4200 rows = 16 blocks + 104), V = 300."""
    check(*setup(4200, 8192, 300, seed=25))


@pytest.mark.parametrize("N", [2048, 2304, 3000])
def test_dz_tile_threshold(N):
    """Kept-row counts around the switch of the dZ producer to 256-row tiles
    (at 2304 rows), with the entropy term."""
    check(*setup(N, 128, 900, seed=29))


def test_wide_tile_dz_producer():
    """>= 2304 kept rows: the dZ producer runs 256-row tiles (4500 rows =
    17 blocks + 148), with the entropy term and temperature."""
    check(*setup(4500, 128, 1500, seed=14), inv_temp=1.0 / 0.9)


def test_wide_tile_dz_tiny_vocabulary_single_k_block():
    """dZ on 256-row tiles with V = 17 (a 17-column store box, clipped by the
    tensor map) and d = 64 (one k-block per tile)."""
    check(*setup(4500, 64, 17, seed=17))


def test_wide_tile_dz_27b_hidden_size():
    """256-row dZ tiles at d = 5120 (80 k-blocks per tile), 4500 rows (a
    ragged last 32-row store box), V = 700 (a 28-column last store box)."""
    check(*setup(4500, 5120, 700, seed=16))


def test_row_chunks_across_the_wide_tile_threshold():
    """A workspace for 4352-row chunks: 9000 rows run as 4352 + 4352 (dZ on
    256-row tiles) + 296 (128-row tiles), grad_w accumulating over chunks."""
    wl, g, ge = setup(9000, 128, 600, seed=15)
    check(wl, g, ge, rows_per_chunk=4352)


def test_wide_tile_grad_hidden_long_vocabulary():
    """K = V >= 64 k-blocks: grad_hidden runs 256-row tiles (600 rows =
    2 blocks + 88, vocabulary tail of 33 columns)."""
    check(*setup(600, 256, 16481, seed=10))


def test_wide_tile_grad_w_many_rows_with_accumulate():
    """K = rows >= 64 k-blocks: grad_w runs 256-row vocabulary tiles
    (V = 700 = 2 blocks + 188) over 16,500 rows, accumulating."""
    wl, g, ge = setup(16500, 128, 700, seed=11)
    base = torch.randn(700, 128, generator=torch.Generator().manual_seed(12))
    check(wl, g, ge, accumulate_base=base)


@pytest.mark.parametrize("N", [4032, 4096, 4100])
def test_grad_w_tile_threshold(N):
    """grad_w's K (kept rows) around the switch to 256-row tiles at 64
    k-blocks: 63 blocks, exactly 64, and 64 plus a 4-row tail block."""
    check(*setup(N, 64, 500, seed=30))


@pytest.mark.parametrize("V", [4032, 4097])
def test_grad_hidden_tile_threshold(V):
    """grad_hidden's K (the vocabulary) on both sides of 64 k-blocks."""
    check(*setup(300, 128, V, seed=31))


def test_wide_tile_with_short_device_count():
    """The host sizes grad_w for all 16,500 rows (wide tiles); the keep-mask
    leaves ~1/3 of them, so the device-side K is far shorter."""
    wl, g, _ = setup(16500, 128, 700, seed=13)
    g[np.arange(16500) % 3 != 0] = 0.0
    out, _ = check(wl, g, None)
    assert torch.count_nonzero(out["grad_hidden"][1::3]) == 0


def test_peaked_softmax():
    check(*setup(256, 256, 2048, seed=6, w_scale=8.0))


def test_extreme_logits():
    """W x 64: the softmax is nearly one-hot, dZ nearly g (1[v = y] - 1[v = argmax])."""
    check(*setup(300, 128, 1500, seed=18, w_scale=64.0))


@pytest.mark.parametrize("N", [450, 4500])  # 128-row and 256-row dZ tiles
def test_deterministic_bitwise(N):
    """No atomics, fixed reduction orders: two calls give identical bits."""
    wl, g, ge = setup(N, 128, 1000, seed=19)
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    fw = mc.token_logprobs(h, w, y)
    a = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g.cuda(), ge.cuda())
    b = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g.cuda(), ge.cuda())
    assert torch.equal(a["grad_hidden"], b["grad_hidden"]) and torch.equal(a["grad_w"], b["grad_w"])


def test_row_keep_gate_equals_zeroed_upstream():
    """row_keep = 0 on a dropped sequence gives the same gradients as zeroing
    its upstream gradient (the M_i factor of Eq. 17)."""
    wl, g, ge = setup(384, 128, 1500, seed=7)
    keep = torch.ones(384, dtype=torch.uint8)
    keep[100:260] = 0
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    fw = mc.token_logprobs(h, w, y)
    a = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g.cuda(), ge.cuda(), row_keep=keep.cuda())
    g0, ge0 = g * keep.float(), ge * keep.float()
    b = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g0.cuda(), ge0.cuda())
    assert torch.equal(a["grad_hidden"], b["grad_hidden"])
    assert torch.equal(a["grad_w"], b["grad_w"])
    ref = oracle.token_logprobs_bwd(wl.hidden, wl.w_vocab, wl.targets, g0, ge0)
    assert rel_fro(np_(a["grad_w"]), ref["grad_w"]) <= TOL_GRAD


@pytest.mark.parametrize("N", [300, 16500])  # grad_w on 128-row and on 256-row tiles (K >= 4096)
def test_every_row_dropped(N):
    """row_keep all 0: no row has a gradient, so the device-side K of grad_w is
    0: grad_hidden and grad_w are zero, or grad_w keeps its value when
    accumulating."""
    wl, g, ge = setup(N, 64, 300, seed=20)
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    fw = mc.token_logprobs(h, w, y)
    keep = torch.zeros(N, dtype=torch.uint8, device="cuda")
    out = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g.cuda(), ge.cuda(), row_keep=keep)
    torch.cuda.synchronize()
    assert not out["grad_hidden"].any() and not out["grad_w"].any()
    base = torch.randn(300, 64, device="cuda")
    gw = base.clone()
    mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g.cuda(), ge.cuda(), row_keep=keep, grad_w=gw,
                          accumulate=True)
    torch.cuda.synchronize()
    assert torch.equal(gw, base)


def test_zero_rows():
    wl, g, _ = setup(8, 64, 300, seed=21)
    h, w, y = wl.hidden.cuda()[:0], wl.w_vocab.cuda(), wl.targets.cuda()[:0]
    z = torch.empty(0, device="cuda")
    out = mc.token_logprobs_bwd(h, w, y, z, None, z)
    torch.cuda.synchronize()
    assert out["grad_hidden"].shape == (0, 64) and not out["grad_w"].any()


def test_out_of_range_targets_are_skipped_and_flagged():
    """Targets outside [0, V) in two different 1,024-row selection slabs: the
    row selection sets MC_DEV_TARGET_RANGE and leaves those rows out (zero
    gradient, their NaN lse never read); every other row matches the oracle
    with those rows' upstream gradient zeroed."""
    wl, g, ge = setup(2100, 64, 700, seed=22)
    y_bad = wl.targets.clone()
    y_bad[5] = 700
    y_bad[1500] = -1
    h, w = wl.hidden.cuda(), wl.w_vocab.cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    fw = mc.token_logprobs(h, w, y_bad.cuda())
    out = mc.token_logprobs_bwd(h, w, y_bad.cuda(), fw["lse"], fw["entropy"], g.cuda(), ge.cuda(), dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & mc.MC_DEV_TARGET_RANGE
    gh = out["grad_hidden"]
    assert not gh[5].any() and not gh[1500].any()
    g0, ge0 = g.clone(), ge.clone()
    g0[[5, 1500]] = 0.0
    ge0[[5, 1500]] = 0.0
    y_ok = y_bad.clone()
    y_ok[[5, 1500]] = 0
    ref = oracle.token_logprobs_bwd(wl.hidden, wl.w_vocab, y_ok, g0, ge0)
    assert rel_fro(np_(gh.float()), ref["grad_hidden"]) <= TOL_GRAD
    assert rel_fro(np_(out["grad_w"]), ref["grad_w"]) <= TOL_GRAD
