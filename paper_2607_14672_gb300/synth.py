"""Seeded synthetic inputs shared by the tests, the bench and the oracle runs.

This module draws random numbers only; it holds none of the method's
arithmetic. Both the CUDA path and the float64 oracle are fed from here.
All generators use numpy's PCG64 ``default_rng`` and return float64 arrays
(callers cast); silent spikes are +inf.

Workload shapes follow the paper's experiments (App. C, App. E) with
synthetic data standing in for the image datasets, which are not shipped:
  * uniform spike times in [lo, hi) with an independent Bernoulli silent mask
    (the random-input single-layer experiments of Sec. 3, Fig. 2);
  * pixel intensities x ~ U[0, 1) with a fraction set to 0, time-encoded as
    t = tau_in (1 - x) with x = 0 treated as a silent input (App. C.2
    encoding; the silent reading of x = 0 follows the workload definition).
"""

import numpy as np


def rng(seed):
    return np.random.default_rng(seed)


def uniform_spikes(seed, shape, lo=0.0, hi=1.0, silent_frac=0.0):
    """Spike times ~ U[lo, hi), each independently silent with prob silent_frac."""
    g = rng(seed)
    t = g.uniform(lo, hi, size=shape)
    silent = g.random(size=shape) < silent_frac
    return np.where(silent, np.inf, t)


def intensity_spikes(seed, shape, zero_frac=0.0, tau_in=1.0):
    """Image-like input: x ~ U[0,1) with a zero_frac share set to 0, encoded
    as t = tau_in (1 - x); x = 0 gives a silent (+inf) input."""
    g = rng(seed)
    x = g.random(size=shape)
    x = np.where(g.random(size=shape) < zero_frac, 0.0, x)
    return np.where(x > 0.0, tau_in * (1.0 - x), np.inf)


def doubled_intensity_spikes(seed, shape, tau_in=1.0):
    """Colour-image input with the channel doubling of App. C.2: x ~ U[0, 1)
    of shape (B, C, H, W), channels C..2C-1 hold 1 - x, and every pixel is
    encoded as t = tau_in (1 - x) (so no input is silent)."""
    x = rng(seed).random(size=shape)
    x2 = np.concatenate([x, 1.0 - x], axis=1)
    return tau_in * (1.0 - x2)


def normal_weights(seed, shape, mean=0.0, std=1.0):
    return rng(seed).normal(mean, std, size=shape)


def labels(seed, batch, n_classes):
    return rng(seed).integers(0, n_classes, size=batch)


def t_offsets(seed, dts):
    """One t_offset per layer, uniform on (-dt/2, dt/2] (Alg. 2 draws one per layer)."""
    g = rng(seed)
    out = []
    for dt in dts:
        u = g.random()                    # [0, 1)
        out.append(dt / 2.0 - u * dt)     # (-dt/2, dt/2]
    return out
