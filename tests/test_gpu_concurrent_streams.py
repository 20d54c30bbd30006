"""The wave-gated GEMMs (cooperative launches whose CTAs wait on one another
through a bounded counter wait) beside other work on the GPU: the forward and
backward run on one stream while another stream keeps torch matmuls going.
The results are the bits of a run on an idle GPU, and no wait gave up."""

import pytest
import torch

from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def test_gated_kernels_beside_another_stream():
    wl = workloads.build(workloads.spec_for(1, n_seqs=24, len_lo=300, len_hi=700, d=512, V=8192), "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    g = torch.randn(wl.N, device="cuda")

    def run(stream):
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        with torch.cuda.stream(stream):
            fw = mc.token_logprobs(h, w, y, dev_status=st, stream=stream)
            bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g, None, dev_status=st, stream=stream)
        return fw, bw, st

    s1 = torch.cuda.Stream()
    ref_fw, ref_bw, ref_st = run(s1)
    torch.cuda.synchronize()
    assert int(ref_st.item()) == 0

    s2 = torch.cuda.Stream()
    a = torch.randn(4096, 4096, device="cuda", dtype=torch.bfloat16)
    with torch.cuda.stream(s2):
        for _ in range(60):
            a = torch.matmul(a, a).clamp_(-1, 1)
    got_fw, got_bw, got_st = run(s1)
    torch.cuda.synchronize()
    assert int(got_st.item()) == 0, "a bounded wait gave up"
    for k in ("logp", "entropy", "lse"):
        assert torch.equal(got_fw[k], ref_fw[k]), k
    assert torch.equal(got_bw["grad_hidden"], ref_bw["grad_hidden"])
    assert torch.equal(got_bw["grad_w"], ref_bw["grad_w"])
