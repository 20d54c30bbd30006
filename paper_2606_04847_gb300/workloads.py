"""Seeded synthetic workloads for the log-prob / MirrorPop hot path.

This module only draws inputs. It holds none of the hot path's arithmetic (no
log-softmax, entropy, ratio statistics, mask or gradient); the oracle and the
CUDA path both take their inputs from here and nothing else is shared between
them. The one model-shaped computation here is the rollout stand-in that draws
each target token from the softmax of the generator's own logits (Gumbel-max
sampling); only the sampled indices leave it.

The paper's workloads are Qwen3.5-9B / Qwen3.6-27B RL rollouts on kernel-
generation prompts (§5.1). Neither the weights nor the prompts exist here, so
these seeded inputs with the same shapes stand in for them:

=====  =====================================================  =====  ======
config sequences / tokens                                      d      V
=====  =====================================================  =====  ======
1      8 x 32 (N = 256)                                        512    4096
2      16 x 2048 (N = 32768)                                   4096   151936
3      32, lengths U{512..8192}, padded then packed            4096   248320
4      64 multi-turn, lengths U{1024..16384}, per-turn mask    5120   248320
5      config 3 + per-token advantage weights (backward)       4096   248320
=====  =====================================================  =====  ======

Values: hidden ~ N(0, 1) and W_vocab ~ N(0, (1/sqrt(d))^2), both rounded to
bf16 (round-to-nearest-even), so logits have a standard deviation near 1.
Targets: uniform in [0, V) (config 1) or sampled from softmax(z / tau) at
tau = 1 (configs 2-5). Behaviour log-probs are the policy's log-probs plus the
``gap`` drawn here (logp_behaviour = logp_policy_reference + gap):
  config 1: N(0, 0.05^2) per token;
  config 2: N(0, 0.1^2) per token on a seeded 10 % of the sequences, 0 elsewhere;
  configs 3-5: one N(0, 0.2^2) draw per sequence, added to all its tokens.
Config 5 adds advantage weights a_t ~ N(0, 1); the backward's upstream
gradient is g_t = a_t * keep_{seq(t)} * loss_mask_t.

Each tensor comes from its own generator seeded from (config seed, name), so
changing one tensor's recipe does not move the others. The CPU generator gives
the same bits on every machine; the CUDA generator is used for full-size inputs
(fast) and is reproducible on a given GPU type.
"""

from __future__ import annotations

import dataclasses
import hashlib
import math
from typing import Optional, Sequence

import torch

__all__ = ["WorkloadSpec", "Workload", "CONFIGS", "spec_for", "build", "cancellation_gap"]


@dataclasses.dataclass(frozen=True)
class WorkloadSpec:
    name: str
    seed: int
    n_seqs: int
    len_lo: int                  # sequence length drawn uniformly in [len_lo, len_hi]
    len_hi: int
    d: int
    V: int
    targets: str                 # "uniform" | "sampled"
    gap: str                     # "token" | "token_subset" | "sequence"
    gap_std: float
    gap_frac: float = 1.0        # fraction of sequences perturbed ("token_subset")
    multi_turn: bool = False
    advantages: bool = False
    inv_temperature: float = 1.0
    sample_inv_temperature: float = 1.0
    delta: float = 0.2
    w_scale: float = 1.0         # multiplies W's std (>1: peaked softmax)
    padded: bool = False         # lengths vary: generated padded [B, max L], then packed


CONFIGS = {
    1: WorkloadSpec("tiny-fwd N=256 d=512 V=4096", 0, 8, 32, 32, 512, 4096,
                    "uniform", "token", 0.05, delta=0.04),
    2: WorkloadSpec("mid-fwd 16x2048 d=4096 V=151936", 1, 16, 2048, 2048, 4096, 151936,
                    "sampled", "token_subset", 0.1, gap_frac=0.1, delta=0.05),
    3: WorkloadSpec("9B-class-fwd 32 seqs L~U[512,8192] d=4096 V=248320", 2, 32, 512, 8192,
                    4096, 248320, "sampled", "sequence", 0.2, delta=0.2, padded=True),
    4: WorkloadSpec("27B-class-fwd 64 multi-turn seqs L~U[1024,16384] d=5120 V=248320", 3, 64,
                    1024, 16384, 5120, 248320, "sampled", "sequence", 0.2, multi_turn=True,
                    delta=0.2, padded=True),
    5: WorkloadSpec("9B-class-fwd+bwd 32 seqs L~U[512,8192] d=4096 V=248320", 4, 32, 512, 8192,
                    4096, 248320, "sampled", "sequence", 0.2, advantages=True, delta=0.2,
                    padded=True),
}


def spec_for(config: int, **overrides) -> WorkloadSpec:
    """The spec of a config, optionally with fields replaced (e.g. smaller shapes)."""
    return dataclasses.replace(CONFIGS[config], **overrides)


@dataclasses.dataclass
class Workload:
    spec: WorkloadSpec
    hidden: torch.Tensor         # bf16 [N, d]
    w_vocab: torch.Tensor        # bf16 [V, d]
    targets: torch.Tensor        # int32 [N]
    cu_seqlens: torch.Tensor     # int64 [B+1]
    loss_mask: torch.Tensor      # uint8 [N]
    gap: torch.Tensor            # fp32 [N]: logp_behaviour - logp_policy_reference
    advantages: Optional[torch.Tensor]  # fp32 [N] or None
    seq_lens: list
    max_len: int

    @property
    def N(self) -> int:
        return self.hidden.shape[0]

    @property
    def B(self) -> int:
        return self.cu_seqlens.shape[0] - 1


def _seed(base: int, name: str) -> int:
    h = hashlib.sha256(f"{base}:{name}".encode()).digest()
    return int.from_bytes(h[:8], "little") & ((1 << 63) - 1)


def _gen(device, base: int, name: str) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(_seed(base, name))
    return g


def _lengths(spec: WorkloadSpec, lengths: Optional[Sequence[int]]):
    if lengths is not None:
        return [int(x) for x in lengths]
    g = _gen("cpu", spec.seed, "lengths")
    if spec.len_lo == spec.len_hi:
        return [spec.len_lo] * spec.n_seqs
    return torch.randint(spec.len_lo, spec.len_hi + 1, (spec.n_seqs,), generator=g).tolist()


def _turn_mask(spec: WorkloadSpec, lens, first_turn_only: bool) -> torch.Tensor:
    """Per-turn loss mask: each sequence is 1 + U{1,2,3} turns cut at seeded points;
    the first 30 % of each turn is prompt (mask 0), the rest response (mask 1)."""
    g = _gen("cpu", spec.seed, "turns")
    parts = []
    for L in lens:
        n_turns = 1 + int(torch.randint(1, 4, (1,), generator=g))
        n_turns = max(1, min(n_turns, L))
        if n_turns > 1:
            cuts = torch.randperm(L - 1, generator=g)[: n_turns - 1] + 1
            bounds = [0] + sorted(cuts.tolist()) + [L]
        else:
            bounds = [0, L]
        m = torch.zeros(L, dtype=torch.uint8)
        for k in range(len(bounds) - 1):
            a, b = bounds[k], bounds[k + 1]
            if first_turn_only and k > 0:
                break
            p = int(math.floor(0.3 * (b - a)))
            m[a + p: b] = 1
        parts.append(m)
    return torch.cat(parts) if parts else torch.zeros(0, dtype=torch.uint8)


def _sample_targets(hidden, w_vocab, inv_temp, device, seed, rows_per_chunk=1024):
    """Rollout stand-in: y_t ~ softmax(z_t * inv_temp) by Gumbel-max over the
    generator's own logits (fp32 on CPU; bf16 matmul on CUDA)."""
    N = hidden.shape[0]
    V = w_vocab.shape[0]
    out = torch.empty(N, dtype=torch.int32, device=device)
    g = _gen(device, seed, "gumbel")
    wt = w_vocab.t() if device != "cpu" else w_vocab.float().t()
    for r0 in range(0, N, rows_per_chunk):
        r1 = min(N, r0 + rows_per_chunk)
        hb = hidden[r0:r1] if device != "cpu" else hidden[r0:r1].float()
        z = (hb @ wt).float().mul_(inv_temp)
        u = torch.rand((r1 - r0, V), generator=g, device=device).clamp_(min=1e-20)
        z.sub_(u.log_().neg_().log_())           # + Gumbel noise -log(-log u)
        out[r0:r1] = z.argmax(dim=1).to(torch.int32)
        del z, u
    return out


def cancellation_gap(wl: "Workload", magnitude: float = 0.3, frac: float = 0.5,
                     run: int = 4) -> torch.Tensor:
    """Gap variant with directional cancellation (§4.5.2 and the cancellation
    appendix): on a seeded ``frac`` of the sequences the per-token gap alternates
    sign every ``run`` tokens with fixed magnitude, so the signed mean is near 0
    while the absolute mean is ``magnitude``. Other sequences keep ``wl.gap``."""
    g = _gen("cpu", wl.spec.seed, "cancel")
    gap = wl.gap.detach().cpu().clone()
    B = wl.B
    cu = wl.cu_seqlens.cpu().tolist()
    chosen = torch.randperm(B, generator=g)[: int(round(frac * B))].tolist()
    for i in chosen:
        L = cu[i + 1] - cu[i]
        sign = torch.tensor([1.0 if (k // run) % 2 == 0 else -1.0 for k in range(L)])
        gap[cu[i]: cu[i + 1]] = magnitude * sign
    return gap.to(wl.gap.device)


def build(spec: WorkloadSpec, device="cpu", lengths: Optional[Sequence[int]] = None,
          first_turn_only: bool = False) -> Workload:
    """Draw one workload. ``lengths`` overrides the seeded sequence lengths
    (zero-length sequences allowed)."""
    device = str(device)
    lens = _lengths(spec, lengths)
    N = int(sum(lens))
    B = len(lens)
    d, V = spec.d, spec.V
    cu = torch.zeros(B + 1, dtype=torch.int64)
    if B:
        cu[1:] = torch.cumsum(torch.tensor(lens, dtype=torch.int64), 0)

    hidden = torch.randn((N, d), generator=_gen(device, spec.seed, "hidden"),
                         device=device, dtype=torch.float32).to(torch.bfloat16)
    w = torch.randn((V, d), generator=_gen(device, spec.seed, "w_vocab"),
                    device=device, dtype=torch.float32)
    w.mul_(spec.w_scale / math.sqrt(d))
    w_vocab = w.to(torch.bfloat16)
    del w

    if spec.targets == "uniform":
        targets = torch.randint(0, V, (N,), generator=_gen("cpu", spec.seed, "targets"),
                                dtype=torch.int64).to(torch.int32).to(device)
    else:
        targets = _sample_targets(hidden, w_vocab, spec.sample_inv_temperature, device,
                                  spec.seed)

    if spec.multi_turn:
        loss_mask = _turn_mask(spec, lens, first_turn_only)
    else:
        loss_mask = torch.ones(N, dtype=torch.uint8)

    gg = _gen("cpu", spec.seed, "gap")
    if spec.gap == "token":
        gap = torch.randn(N, generator=gg) * spec.gap_std
    elif spec.gap == "token_subset":
        gap = torch.zeros(N)
        k = max(1, int(math.ceil(spec.gap_frac * B))) if B else 0
        for i in torch.randperm(B, generator=gg)[:k].tolist():
            gap[cu[i]: cu[i + 1]] = torch.randn(lens[i], generator=gg) * spec.gap_std
    else:  # "sequence"
        per_seq = torch.randn(B, generator=gg) * spec.gap_std
        gap = torch.repeat_interleave(per_seq, torch.tensor(lens, dtype=torch.int64)) \
            if B else torch.zeros(0)

    adv = None
    if spec.advantages:
        adv = torch.randn(N, generator=_gen("cpu", spec.seed, "advantages")).to(device)

    return Workload(spec=spec, hidden=hidden, w_vocab=w_vocab, targets=targets,
                    cu_seqlens=cu.to(device), loss_mask=loss_mask.to(device),
                    gap=gap.float().to(device), advantages=adv, seq_lens=lens,
                    max_len=max(lens) if lens else 0)
