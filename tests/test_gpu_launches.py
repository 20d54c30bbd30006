"""Kernels per call, from libmc's own launch counter (mc_kernel_launches):
the forward is the projection + log-softmax engine and one finalize kernel,
the filter one kernel, the backward a three-pass row selection, a gather and
three GEMM engines per row chunk (plus one status merge when the caller asks
for a status word). No other kernel runs behind these calls."""

import pytest
import torch

from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def _delta(fn):
    torch.cuda.synchronize()
    before = mc.kernel_launches()
    fn()
    torch.cuda.synchronize()
    return mc.kernel_launches() - before


def test_kernels_per_call():
    wl = workloads.build(workloads.spec_for(1, n_seqs=3, len_lo=300, len_hi=300, d=128, V=1000), "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    fw = mc.token_logprobs(h, w, y)
    assert _delta(lambda: mc.token_logprobs(h, w, y, out=fw)) == 2
    lb = (fw["logp"] + wl.gap.cuda()).contiguous()
    cu = wl.cu_seqlens.cuda()
    assert _delta(lambda: mc.seq_ratio_filter(fw["logp"], lb, None, cu, 0.04, 0.04)) == 1
    g = torch.randn(wl.N, device="cuda")
    bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g)
    args = (h, w, y, fw["lse"], fw["entropy"], g)
    kw = dict(grad_hidden=bw["grad_hidden"], grad_w=bw["grad_w"])
    assert _delta(lambda: mc.token_logprobs_bwd(*args, **kw)) == 3 + 1 + 3
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert _delta(lambda: mc.token_logprobs_bwd(*args, dev_status=st, **kw)) == 3 + 1 + 3 + 1
    # 900 rows in chunks of 256: four chunks of three GEMM launches each.
    assert _delta(lambda: mc.token_logprobs_bwd(*args, rows_per_chunk=256, **kw)) == 3 + 1 + 3 * 4
