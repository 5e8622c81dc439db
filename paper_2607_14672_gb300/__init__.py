"""GB300-native DSTD training of TTFS LIF layers (differentiable spike-time
discretization, arxiv 2607.14672).

The compute path is ``libdstd.so`` (hand-written sm_103a CUDA behind a C-ABI,
``include/dstd.h``); ``dstd`` is its thin Python binding and ``net`` a
multi-layer driver over it. ``synth`` and ``configs`` define the seeded
synthetic workloads.
"""

__all__ = ["synth", "configs"]
