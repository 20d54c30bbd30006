"""The C-ABI library loads, exports every symbol include/mc.h declares, and
rejects bad arguments on the host with the documented codes (no GPU needed:
these calls return before any CUDA call)."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mc.h")

INVALID, UNSUPPORTED, CUDA, WORKSPACE = 1, 2, 3, 5


@pytest.fixture(scope="module")
def L():
    from paper_2606_04847_gb300 import build, mc

    if not os.path.exists(mc.lib_path()):
        build.build()
    return mc.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(mc_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for f in ("mc_token_logprobs", "mc_token_logprobs_bwd", "mc_seq_ratio_filter",
              "mc_token_logprobs_workspace_size", "mc_token_logprobs_bwd_workspace_size"):
        assert f in names


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name


def test_binding_signatures_match_header(L):
    from paper_2606_04847_gb300 import mc

    assert sorted(mc.SIGNATURES) == declared_functions()


def test_version_and_status_strings(L):
    assert L.mc_version() >> 16 == 1
    for code in range(7):
        assert L.mc_status_string(code).decode().startswith("MC_")
    assert L.mc_last_cuda_error() is not None


def test_workspace_queries(L):
    fw = L.mc_token_logprobs_workspace_size(256, 512, 4096)
    assert fw >= 256 + 3 * 16 * 256 * 4 + 256 * 4 and fw % 256 == 0
    assert L.mc_token_logprobs_workspace_size(256, 100, 4096) == 0  # d % 64 != 0
    one_chunk = L.mc_token_logprobs_bwd_workspace_size(1000, 512, 4097, 1000)
    assert one_chunk >= 1024 * 4160 * 2  # rows padded to 128, V padded to 64, bf16
    small = L.mc_token_logprobs_bwd_workspace_size(1000, 512, 4097, 128)
    assert 128 * 4160 * 2 <= small < one_chunk
    assert L.mc_token_logprobs_bwd_workspace_size(10, 512, 4096, 0) == 0


FAKE = 0x10000  # aligned non-null stand-in pointer; never dereferenced by these calls


def fwd(L, hidden=FAKE, w=FAKE, targets=FAKE, N=256, d=512, V=4096, inv_t=1.0, logp=FAKE, ws=FAKE,
        ws_bytes=1 << 30):
    return L.mc_token_logprobs(hidden, w, targets, N, d, V, inv_t, logp, None, None, ws, ws_bytes, None, None)


def test_forward_argument_checks(L):
    assert fwd(L, N=-1) == INVALID
    assert fwd(L, d=100) == INVALID
    assert fwd(L, d=0) == INVALID
    assert fwd(L, V=0) == INVALID
    assert fwd(L, inv_t=0.0) == INVALID
    assert fwd(L, inv_t=float("inf")) == INVALID
    assert fwd(L, hidden=None) == INVALID
    assert fwd(L, logp=None) == INVALID
    assert fwd(L, hidden=FAKE + 2) == INVALID  # not 16-byte aligned
    assert fwd(L, ws=None) == WORKSPACE
    assert fwd(L, ws=FAKE + 16) == WORKSPACE  # not 256-byte aligned
    assert fwd(L, ws_bytes=100) == WORKSPACE
    assert fwd(L, N=0) == 0  # nothing to do


def test_host_detected_errors_queue_no_kernels(L):
    """Calls rejected on the host (bad sizes, pointers, workspaces) launch
    nothing: the library's launch counter does not move."""
    before = L.mc_kernel_launches()
    assert fwd(L, N=-1) == INVALID
    assert fwd(L, d=100) == INVALID
    assert fwd(L, ws=None) == WORKSPACE
    assert fwd(L, N=0) == 0
    assert bwd(L, d=100) == INVALID
    assert bwd(L, ws_bytes=100) == WORKSPACE
    assert L.mc_kernel_launches() == before


def test_forward_without_gpu_reports_device_error(L):
    import torch

    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    assert fwd(L) in (CUDA, UNSUPPORTED)


def bwd(L, N=256, d=512, V=4096, ws_bytes=1 << 30, grad_w=FAKE, grad_entropy=None, entropy=None):
    return L.mc_token_logprobs_bwd(FAKE, FAKE, FAKE, FAKE, entropy, FAKE, grad_entropy, None, N, d, V, 1.0, FAKE,
                                   grad_w, 0, FAKE, ws_bytes, None, None)


def test_backward_argument_checks(L):
    assert bwd(L, d=96) == INVALID
    assert bwd(L, grad_w=None) == INVALID
    assert bwd(L, grad_entropy=FAKE, entropy=None) == INVALID
    assert bwd(L, ws_bytes=1000) == WORKSPACE


def filt(L, B=2, N=10, delta=0.1, cu=FAKE, keep=FAKE, lp=FAKE):
    return L.mc_seq_ratio_filter(lp, FAKE, None, cu, B, N, delta, -1.0, FAKE, FAKE, FAKE, keep, None, None,
                                 None, None)


def test_filter_argument_checks(L):
    assert filt(L, B=0) == INVALID
    assert filt(L, N=-1) == INVALID
    assert filt(L, delta=-0.1) == INVALID
    assert filt(L, delta=float("nan")) == INVALID
    assert filt(L, cu=None) == INVALID
    assert filt(L, keep=None) == INVALID
    assert filt(L, lp=None) == INVALID
    assert filt(L, cu=FAKE + 4) == INVALID  # int64 array not 8-byte aligned


def loss_call(L, B=2, N=10, eps_low=0.2, eps_high=0.2, keep=FAKE, ws=FAKE, ws_bytes=1 << 20, beta=0.0,
              ref=None):
    return L.mc_grpo_masked_loss(FAKE, FAKE, None, FAKE, FAKE, keep, FAKE, B, N, eps_low, eps_high, ref, beta,
                                 FAKE, FAKE, None, None, None, ws, ws_bytes, None)


def test_loss_argument_checks(L):
    assert L.mc_grpo_masked_loss_workspace_size(0) == 0
    assert L.mc_grpo_masked_loss_workspace_size(1000) >= 256 + 4000
    assert loss_call(L, B=0) == INVALID
    assert loss_call(L, eps_low=1.0) == INVALID
    assert loss_call(L, eps_low=-0.1) == INVALID
    assert loss_call(L, eps_high=float("inf")) == INVALID
    assert loss_call(L, keep=None) == INVALID
    assert loss_call(L, beta=-1.0) == INVALID
    assert loss_call(L, beta=float("nan")) == INVALID
    assert loss_call(L, ref=FAKE + 2) == INVALID  # misaligned reference log-probs
    assert loss_call(L, ws=None) == WORKSPACE
    assert loss_call(L, ws_bytes=16) == WORKSPACE


def adv_call(L, T=16, K=3, G=8, alpha=0.75, eps=1e-6, adv=FAKE):
    return L.mc_prime_echo_advantages(FAKE, FAKE, FAKE, T, K, G, alpha, 0.5, 0.2, eps, None, adv, None)


def test_advantage_argument_checks(L):
    assert adv_call(L, T=10, G=8) == INVALID  # T not a multiple of the group size
    assert adv_call(L, K=0) == INVALID
    assert adv_call(L, G=0) == INVALID
    assert adv_call(L, alpha=1.5) == INVALID
    assert adv_call(L, eps=-1.0) == INVALID
    assert adv_call(L, adv=None) == INVALID


def test_shard_argument_checks(L):
    def state(v_begin=0, st=FAKE, d=64):
        return L.mc_token_logprob_state(FAKE, FAKE, FAKE, 16, d, 100, v_begin, 1.0, st, FAKE, 1 << 20, None, None)

    assert state(v_begin=-1) == INVALID
    assert state(st=None) == INVALID
    assert state(st=FAKE + 4) == INVALID  # state rows are float4: 16-byte alignment
    assert state(d=65) == INVALID
    assert L.mc_merge_logprob_states(FAKE, 0, 16, FAKE, None, None, None, None) == INVALID
    assert L.mc_merge_logprob_states(FAKE + 8, 2, 16, FAKE, None, None, None, None) == INVALID
    assert L.mc_merge_logprob_states(FAKE, 2, 0, FAKE, None, None, None, None) == 0


def test_selftest_argument_checks(L):
    assert L.mc_selftest_bounded_wait(None, 10 ** 8, None) == INVALID
    assert L.mc_selftest_bounded_wait(FAKE, 10, None) == INVALID
    assert L.mc_selftest_bounded_wait(FAKE, 10 ** 12, None) == INVALID


def test_binding_fails_loudly_without_cuda_tensors(L):
    import torch

    from paper_2606_04847_gb300 import mc

    h = torch.zeros(4, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        mc.token_logprobs(h, h, torch.zeros(4, dtype=torch.int32))
