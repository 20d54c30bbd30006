"""The CTA-pair engine (tcgen05 cta_group::2, selected with MC_ENGINE=pair)
against the fp64 oracle: forward on the tiny config and a ragged shape, and
the backward on a ragged shape with two row chunks. The engine is chosen once
per process, so the checks run in a child process."""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys
sys.path.insert(0, {root!r}); sys.path.insert(0, {tests!r})
import numpy as np, torch
import oracle
from gpu_util import TOL_LOGP, TOL_ENT, TOL_GRAD, assert_close_abs, np_, rel_fro
from paper_2606_04847_gb300 import mc, workloads

for spec in (workloads.spec_for(1), workloads.spec_for(1, n_seqs=1, len_lo=300, len_hi=300, d=128, V=4097)):
    wl = workloads.build(spec, "cpu")
    out = mc.token_logprobs(wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda())
    ref = oracle.token_logprobs(wl.hidden, wl.w_vocab, wl.targets)
    assert_close_abs(np_(out["logp"]), ref["logp"], TOL_LOGP, "logp")
    assert_close_abs(np_(out["entropy"]), ref["entropy"], TOL_ENT, "entropy")

spec = workloads.spec_for(1, n_seqs=1, len_lo=450, len_hi=450, d=128, V=700, seed=3)
wl = workloads.build(spec, "cpu")
g = torch.randn(450, generator=torch.Generator().manual_seed(1))
ge = torch.randn(450, generator=torch.Generator().manual_seed(2)) * 0.3
h, w, y = wl.hidden.cuda(), wl.w_vocab.cuda(), wl.targets.cuda()
fw = mc.token_logprobs(h, w, y)
bw = mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], g.cuda(), ge.cuda(), rows_per_chunk=256)
torch.cuda.synchronize()
ref = oracle.token_logprobs_bwd(wl.hidden, wl.w_vocab, wl.targets, g, ge)
assert rel_fro(np_(bw["grad_hidden"].float()), ref["grad_hidden"]) <= TOL_GRAD
assert rel_fro(np_(bw["grad_w"]), ref["grad_w"]) <= TOL_GRAD
print("pair engine ok")
"""


def test_pair_engine_parity():
    code = CHILD.format(root=ROOT, tests=os.path.join(ROOT, "tests"))
    env = dict(os.environ, MC_ENGINE="pair", MC_WAIT_TIMEOUT_NS="2000000000")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "pair engine ok" in r.stdout
