"""CPU fp64 oracle for the fused log-prob / MirrorPop hot path.

This package is TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU-baseline / reference leg may import it. The product path
(the C-ABI library and its Python binding) never imports, links or calls it, and
it shares no code with the CUDA kernels: it is the plain, slow, two-pass
definition of what the kernels compute, written in NumPy float64 so that a
reader can check it against the paper by eye.

Modules
-------
``oracle.logprobs``  per-token target log-prob, entropy and log-sum-exp of the
                     LM-head softmax, and its closed-form backward.
``oracle.filter``    per-sequence signed / absolute mean log importance ratio,
                     the MirrorPop keep-mask (Eq. 18-21, §4.5.2) and per-token
                     ratios (Eq. 4).
``oracle.grpo``      the masked GRPO clipped-surrogate loss (Eq. 5 / Eq. 17,
                     without the KL term) and its gradient.
``oracle.advantage`` the PrimeEcho trajectory reward (Eq. 9-10) and the
                     group-normalised advantage (Eq. 12 / Eq. 3).

Every function names the passage it follows. Parity is pinned for every
function by the ``-m "not gpu"`` tests in ``tests/test_oracle_*.py`` (brute
force, closed forms, invariants, library routines, finite differences and the
paper's worked example); none is "parity unpinned".
"""

from .logprobs import logprob_state, token_logprobs, token_logprobs_bwd, token_logprobs_bwd_rows  # noqa: F401
from .filter import seq_ratio_filter  # noqa: F401
from .grpo import grpo_masked_loss  # noqa: F401
from .advantage import group_advantage, prime_echo_reward  # noqa: F401
