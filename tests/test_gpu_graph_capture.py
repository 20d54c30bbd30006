"""The step's calls captured in a CUDA graph and replayed give the bits of
the eager calls. The forward's projection is a cooperative launch with a
wave gate; ~12,000 rows give it several waves of units."""

import pytest
import torch

from paper_2606_04847_gb300 import mc, workloads

pytestmark = pytest.mark.gpu


def test_graph_replay_matches_eager():
    wl = workloads.build(workloads.spec_for(1, n_seqs=40, len_lo=200, len_hi=400, d=256, V=3000), "cpu")
    h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
    cu, lb = wl.cu_seqlens.cuda(), torch.randn(wl.N, device="cuda") * 0.05 - 8.0
    g = torch.randn(wl.N, device="cuda")
    N, d, V = wl.N, w.shape[1], w.shape[0]
    fw = {k: torch.empty(N, device="cuda") for k in ("logp", "entropy", "lse")}
    fws = torch.empty(mc.forward_workspace_size(N, d, V), dtype=torch.uint8, device="cuda")
    bws = torch.empty(mc.backward_workspace_size(N, d, V), dtype=torch.uint8, device="cuda")
    gh = torch.empty((N, d), dtype=torch.bfloat16, device="cuda")
    gw = torch.empty((V, d), dtype=torch.float32, device="cuda")

    def step(s):
        mc.token_logprobs(h, w, y, out=fw, workspace=fws, stream=s)
        f = mc.seq_ratio_filter(fw["logp"], lb, None, cu, 0.5, 0.5, stream=s)
        mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g, None, row_keep=f["token_keep"],
                              grad_hidden=gh, grad_w=gw, workspace=bws, stream=s)
        return f

    f = step(torch.cuda.current_stream())
    torch.cuda.synchronize()
    eager = ({k: v.clone() for k, v in fw.items()}, f["keep"].clone(), gh.clone(), gw.clone())
    for t in (*fw.values(), gh, gw):
        t.zero_()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        fg = step(torch.cuda.current_stream())
    for _ in range(2):
        graph.replay()
    torch.cuda.synchronize()
    for k in fw:
        assert torch.equal(fw[k], eager[0][k]), k
    assert torch.equal(fg["keep"], eager[1])
    assert torch.equal(gh, eager[2]) and torch.equal(gw, eager[3])
