"""Vocabulary-sharded forward (mc_token_logprob_state + mc_merge_logprob_states)
vs the unsharded forward and the fp64 oracle: uneven slices (one of a single
column, one smaller than a tile), slice states against the oracle's, the
9B-class vocabulary split as a 4-way tensor-parallel LM head, and a target no
slice holds."""

import numpy as np
import pytest
import torch

import oracle
from gpu_util import TOL_ENT, TOL_LOGP, assert_close_abs, np_
from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def run_shards(h, w, y, bounds, inv_temp=1.0):
    states = torch.empty((len(bounds) - 1, h.shape[0], 4), dtype=torch.float32, device="cuda")
    for p, (a, b) in enumerate(zip(bounds[:-1], bounds[1:])):
        mc.token_logprob_state(h, w[a:b].contiguous(), y, a, inv_temp, state=states[p])
    return states, mc.merge_logprob_states(states)


@pytest.mark.parametrize("N", [300, 4200])  # 128-row and 256-row tiles
def test_uneven_slices_match_unsharded_and_oracle(N):
    spec = workloads.spec_for(1, n_seqs=1, len_lo=N, len_hi=N, d=256, V=4097)
    wl = workloads.build(spec, "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    bounds = [0, 1000, 1001, 1100, 4097]
    states, merged = run_shards(h, w, y, bounds, 1.0 / 0.9)
    full = mc.token_logprobs(h, w, y, 1.0 / 0.9)
    torch.cuda.synchronize()
    for k in ("logp", "entropy", "lse"):
        assert_close_abs(np_(merged[k]), np_(full[k]), 2e-5, f"merged {k} vs unsharded")
    ref = oracle.token_logprobs(wl.hidden, wl.w_vocab, wl.targets, 1.0 / 0.9)
    assert_close_abs(np_(merged["logp"]), ref["logp"], TOL_LOGP, "logp")
    assert_close_abs(np_(merged["entropy"]), ref["entropy"], TOL_ENT, "entropy")
    # each slice's state against the oracle's definition
    for p, (a, b) in enumerate(zip(bounds[:-1], bounds[1:])):
        rs = oracle.logprob_state(wl.hidden, wl.w_vocab[a:b], wl.targets, a, 1.0 / 0.9)
        got = np_(states[p]).astype(np.float64)
        np.testing.assert_allclose(got[:, 0], rs[:, 0], atol=2e-3)                 # max logit
        np.testing.assert_allclose(np.log(got[:, 1]) + got[:, 0], np.log(rs[:, 1]) + rs[:, 0], atol=2e-3)
        own = np.isfinite(rs[:, 3])
        np.testing.assert_array_equal(np.isfinite(got[:, 3]), own)
        np.testing.assert_allclose(got[own, 3], rs[own, 3], atol=2e-3)


def test_tensor_parallel_split_of_the_9b_vocabulary():
    """V = 248,320 split 4 ways as a TP LM head would be, 2,048 tokens."""
    spec = workloads.spec_for(3, n_seqs=1, len_lo=2048, len_hi=2048)
    wl = workloads.build(spec, "cuda")
    V = spec.V
    bounds = [0, V // 4, V // 2, 3 * V // 4, V]
    _, merged = run_shards(wl.hidden, wl.w_vocab, wl.targets, bounds)
    full = mc.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    torch.cuda.synchronize()
    for k in ("logp", "entropy", "lse"):
        assert_close_abs(np_(merged[k]), np_(full[k]), 5e-5, f"merged {k} vs unsharded")


def test_target_in_no_slice():
    spec = workloads.spec_for(1, n_seqs=1, len_lo=64, len_hi=64, d=64, V=512)
    wl = workloads.build(spec, "cpu")
    h, w = wl.hidden.cuda(), wl.w_vocab.cuda()
    y = wl.targets.clone() % 511  # every other target inside the slice
    y[5] = 511
    states = torch.empty((1, 64, 4), dtype=torch.float32, device="cuda")
    mc.token_logprob_state(h, w[:511].contiguous(), y.cuda(), 0, state=states[0])  # column 511 missing
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = mc.merge_logprob_states(states, dev_status=st)
    torch.cuda.synchronize()
    assert int(st.item()) & mc.MC_DEV_TARGET_RANGE
    lp = np_(out["logp"])
    assert np.isnan(lp[5]) and np.isfinite(np.delete(lp, 5)).all()
