"""Reproduce the frozen weight means of the dense workloads (test infrastructure).

Finds, by bisection with the float64 oracle, the weight mean mu_l for which
80% of layer l's neurons fire at initialisation on the seed-0 input batch
(M = 32, t_offset = 0); layer l sees the previous layer's calibrated output.
Prints the values that the workload definitions freeze (CFG2_MU and
CFG3_MU_TIMES_N). Calls only the oracle and the seeded generators.

    python -m oracle.calibrate_configs
"""

import math

import numpy as np

from oracle import dstd, losses
from paper_2607_14672_gb300 import synth


def _mu_for_fraction(t_in, Z, T, dt, tau_v, tau_I, target=0.8, hi=0.2, iters=30):
    lo = 0.0
    for _ in range(iters):
        mu = 0.5 * (lo + hi)
        f = np.isfinite(dstd.forward_dense(t_in, Z + mu, T, dt, tau_v, tau_I, 1.0)["t"]).mean()
        lo, hi = (mu, hi) if f < target else (lo, mu)
    return hi


def calibrate_cfg2(batch=32):
    sizes = [784, 800, 800, 10]
    t = synth.intensity_spikes(0, (batch, 784), 0.6, 1.0)
    mus = []
    for l in range(1, 4):
        wp = losses.window_params(l, 0.1, 1.0, 0.1, 0.2, 0.2)
        T, dt = dstd.grid(wp["t_first"], wp["t_end"], 32, 0.0)
        Z = synth.normal_weights(1000 + l, (sizes[l], sizes[l - 1]), 0.0, 1.0 / math.sqrt(sizes[l - 1]))
        mu = _mu_for_fraction(t, Z, T, dt, 0.5, 0.25)
        mus.append(mu)
        t = dstd.forward_dense(t, Z + mu, T, dt, 0.5, 0.25, 1.0)["t"]
    return mus


def calibrate_cfg3():
    out = []
    for N, B in ((1024, 8), (4096, 4)):
        t = synth.uniform_spikes(0, (B, N), 0.0, 1.0, 0.1)
        Z = synth.normal_weights(1001, (512, N), 0.0, 1.0 / math.sqrt(N))
        T, dt = dstd.grid(0.0, 1.0, 32, 0.0)
        out.append(_mu_for_fraction(t, Z, T, dt, 0.4, 0.2, hi=0.05) * N)
    return out


if __name__ == "__main__":
    print("CFG2_MU", [round(m, 5) for m in calibrate_cfg2()])
    print("CFG3 mu*N", [round(m, 2) for m in calibrate_cfg3()])
