"""GB300-native fused LM-head log-probs, entropy, MirrorPop filter and backward.

The compute lives in ``libmc.so`` (hand-written sm_103a CUDA behind a C ABI,
declared in ``include/mc.h``). ``paper_2606_04847_gb300.mc`` is the thin Python
binding: argument marshalling only, every step runs in the library's kernels.
Importing this package does not load the library; the first call into ``mc``
does, and fails loudly if it has not been built.
"""

import importlib

__all__ = ["mc", "workloads"]


def __getattr__(name):
    if name in __all__:
        return importlib.import_module(f"{__name__}.{name}")
    raise AttributeError(name)
