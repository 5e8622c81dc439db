"""Float64 CPU oracle for DSTD training of TTFS LIF layers.

TEST INFRASTRUCTURE ONLY. This package is the plain, slow, obviously correct
reference that the CUDA library is checked against. Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may import it;
the library and its Python binding never do, and the oracle imports nothing
from the library. Inputs are shared only through the seeded generators in
``paper_2607_14672_gb300.synth``, which hold none of the method's arithmetic.

Modules
-------
lif      neuron model: spike kernel K (Tab. kernel), brute-force ODE
         integration of Eq. LIF_model_TTFS, per-interval coefficient algebra
         of Tab. spike_timing / Tab. timing_DSTD, closed-form and bracketed
         numeric candidate solvers, Lambert W_0.
exact    exact event-driven spike times (Alg. 1, Eq. timing_exact).
dstd     DSTD grid, kernel K_DSTD (Tab. DSTD_kernels, Eq. DSTD_kernel),
         binning, forward (Alg. 2, Eq. timing_DSTD) and analytic backward.
losses   cross-entropy over softmax(-t/tau_soft), temporal penalty T, dead-
         neuron term Q (Eqs. cost_function, temporal_penalty,
         dead_neuron_penalty), AdamW with doubling warm-up.
network  multi-layer dense / conv networks (Alg. 2 layer loop) forward and
         backward, E_RMSE (App. E).

Every numerical function works in float64. Silent neurons carry +inf.
Parity status of each function is stated in its module header.
"""

from . import lif, exact, dstd, losses, network  # noqa: F401
