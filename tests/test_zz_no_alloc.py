"""mc_token_logprobs_noalloc: the forward for callers that may not allocate
device memory (their host's memory manager owns every allocation, or an
allocation's implicit synchronisation is not acceptable where they run).

It must give exactly the bits the workspace entry point gives (and so agree
with the oracle), call after call, while sharing one fixed scratch array
inside the library, and refuse problems larger than that array before
queueing any work. Named so that pytest collects it
last; it does not depend on any other test having run.
"""

import ctypes

import numpy as np
import pytest
import torch

import oracle
from gpu_util import TOL_ENT, TOL_LOGP, assert_close_abs, np_
from paper_2606_04847_gb300 import mc, workloads

SCRATCH_LIMIT = 7
SCRATCH_BYTES = 32 << 20


def _call_noalloc(h, w, y, out, st):
    L = mc.lib()
    return L.mc_token_logprobs_noalloc(
        ctypes.c_void_p(h.data_ptr()), ctypes.c_void_p(w.data_ptr()), ctypes.c_void_p(y.data_ptr()),
        h.shape[0], h.shape[1], w.shape[0], 1.0, ctypes.c_void_p(out["logp"].data_ptr()),
        ctypes.c_void_p(out["entropy"].data_ptr()), ctypes.c_void_p(out["lse"].data_ptr()),
        ctypes.c_void_p(st.data_ptr()), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _run_both(spec, sample=None):
    """One problem through both entry points; returns (workspace outputs,
    no-allocation outputs, workload)."""
    wl = workloads.build(spec, "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    ref = mc.token_logprobs(h, w, y)
    out = {k: torch.full((wl.N,), float("nan"), device="cuda") for k in ("logp", "entropy", "lse")}
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert _call_noalloc(h, w, y, out, st) == 0
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    return ref, out, wl


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    # Problems of different shapes back to back through the same fixed
    # scratch: each call must give exactly the bits of the workspace entry
    # point (same kernels, same schedule, same scratch layout) and nothing a
    # previous call left in the scratch may leak into the next. The 4,096-row
    # case runs 256-row tiles with two column halves (twice the partial
    # slots); 171,008 rows at d = 64, V = 4096 is the largest request the
    # scratch admits.
    cases = [
        workloads.spec_for(1),                                                      # 256 x 512 x 4096
        workloads.spec_for(1, seed=7, n_seqs=3, len_lo=300, len_hi=300, d=256, V=9000),
        workloads.spec_for(1, seed=8, n_seqs=16, len_lo=256, len_hi=256, d=512, V=4096),   # 4,096 rows
        workloads.spec_for(1, seed=9, n_seqs=1, len_lo=171_008, len_hi=171_008, d=64, V=4096),
        workloads.spec_for(1, seed=10, n_seqs=3, len_lo=300, len_hi=300, d=256, V=9000),
    ]
    for spec in cases:
        ref, out, wl = _run_both(spec)
        for k in ("logp", "entropy", "lse"):
            assert torch.equal(out[k], ref[k]), f"{spec.n_seqs}x{spec.len_lo} d={spec.d} V={spec.V}: {k} differs"
        # And against the oracle, on all rows (or 256 sampled rows of the largest case).
        rows = np.arange(wl.N) if wl.N <= 4096 else np.unique(
            np.concatenate([np.random.default_rng(spec.seed).choice(wl.N, 254, replace=False), [0, wl.N - 1]]))
        tr = torch.from_numpy(rows)
        want = oracle.token_logprobs(wl.hidden[tr], wl.w_vocab, wl.targets[tr])
        assert_close_abs(np_(out["logp"])[rows], want["logp"], TOL_LOGP, "logp vs oracle")
        assert_close_abs(np_(out["entropy"])[rows], want["entropy"], TOL_ENT, "entropy vs oracle")
        assert_close_abs(np_(out["lse"])[rows], want["lse"], TOL_LOGP, "lse vs oracle")


def test_noalloc_rejects_problems_beyond_the_fixed_scratch():
    """Host-side check, before any CUDA call, so it also runs without a GPU."""
    L = mc.lib()
    d, V = 512, 4096
    fake = ctypes.c_void_p(0x10000)  # never touched: the size check comes first
    for N in (400_000, 171_009):
        assert L.mc_token_logprobs_workspace_size(N, d, V) > SCRATCH_BYTES
        st = L.mc_token_logprobs_noalloc(fake, fake, fake, N, d, V, 1.0, fake, None, None, None, None)
        assert st == SCRATCH_LIMIT
    assert b"SCRATCH" in L.mc_status_string(SCRATCH_LIMIT)
    # The largest admitted row count for V >= 4096 (about 171,000, as the header states).
    assert L.mc_token_logprobs_workspace_size(171_008, d, V) <= SCRATCH_BYTES
