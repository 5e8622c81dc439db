"""Reproduce the frozen weight means of the dense workloads (test infrastructure).

Finds, by bisection with the float64 oracle, the weight mean mu_l for which
80% of layer l's neurons fire at initialisation on the seed-0 input batch
(t_offset = 0); layer l sees the previous layer's calibrated output. Prints
the values that the workload definitions freeze (CFG2_MU, CFG3_MU_TIMES_N,
CFG4_MU, CFG5_MU, SYN9_MU, SYN20_MU). Calls only the oracle and the seeded generators.

    python -m oracle.calibrate_configs [2] [3] [4] [5] [syn9] [syn20]
"""

import math

import numpy as np

from oracle import dstd, lif, losses, network
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


def _fired_fraction(what, T, dt, tau_v, tau_I, v_th=1.0):
    """Share of neurons whose v^ reaches v_th on some interval (the interval
    maxima of Tab. timing_DSTD's potential, without solving for the time)."""
    M = T.size - 1
    lo, hi = T[:M], T[1:M + 1]
    c = lif.interval_coeffs(lif.lif_case(tau_v, tau_I), tau_v, tau_I, np.broadcast_to(lo, what.shape), what, T[0])
    return float(np.mean(np.any(lif.interval_peak(c, lo, hi) >= v_th, axis=-1)))


def _bisect(frac, target=0.8, lo=-0.5, hi=0.5, iters=26):
    """mu with frac(mu) ~ target; frac increases with mu. The bracket is
    widened first until it holds the target."""
    for _ in range(12):
        if frac(hi) >= target:
            break
        lo, hi = hi, 2.0 * hi
    for _ in range(12):
        if frac(lo) < target:
            break
        lo, hi = 2.0 * lo, lo
    for _ in range(iters):
        mu = 0.5 * (lo + hi)
        lo, hi = (mu, hi) if frac(mu) < target else (lo, mu)
    return 0.5 * (lo + hi)


def calibrate_conv(cfg, batch, verbose=True):
    """mu_l for a conv stack (configs 4, 5): w^(mu) = w^(Z) + mu w^(ones) by
    linearity of the contraction, so each bisection step only re-evaluates
    the interval maxima; the chosen mu's spike times feed the next layer."""
    t0 = cfg["inputs"](B=batch)
    t = t0
    mus, outs = [], []
    for l, L in enumerate(cfg["layers"], start=1):
        T, dt = dstd.grid(L["t_first"], L["t_end"], L["M"], 0.0)
        tv, ti = L["tau_v"], L["tau_I"]
        B = t.shape[0]
        if L.get("skip") is not None:     # skip-and-delay input: delayed source first along channels
            src, delay = L["skip"]
            t = np.concatenate([(t0 if src < 0 else outs[src]) + delay, t], axis=1)
        if L["kind"] == "conv":
            C, H, Wd = t.shape[1:]
            k = L["W"].shape[2]
            Z = synth.normal_weights(1000 + l, L["W"].shape, 0.0, 1.0 / math.sqrt(C * k * k))
            s = dstd.binning(t.reshape(B, -1), T, dt, tv, ti).reshape(B, L["M"], C, H, Wd)
            A = network.conv_what(s, Z, L["stride"], L["pad"])
            U = network.conv_what(s, np.ones((1,) + Z.shape[1:]), L["stride"], L["pad"])
            shape = A.shape
            A, U = A.reshape(B, -1, L["M"]), U.reshape(B, -1, L["M"])
            Ur = np.broadcast_to(U.reshape(B, 1, -1, L["M"]), (B, shape[1], shape[2] * shape[3], L["M"])).reshape(A.shape)
        else:
            x = t.reshape(B, -1)
            Z = synth.normal_weights(1000 + l, L["W"].shape, 0.0, 1.0 / math.sqrt(x.shape[1]))
            s = dstd.binning(x, T, dt, tv, ti)
            A = np.einsum("bmj,ij->bim", s, Z)
            Ur = np.broadcast_to(np.einsum("bmj->bm", s)[:, None, :], A.shape)
        mu = _bisect(lambda m: _fired_fraction(A + m * Ur, T, dt, tv, ti))
        mus.append(mu)
        ctx = dstd.solve(A + mu * Ur, T, dt, tv, ti, 1.0)
        t = ctx["t"].reshape((B,) + tuple(shape[1:4])) if L["kind"] == "conv" else ctx["t"]
        outs.append(t)
        if verbose:
            print(f"layer {l}: mu {mu:.5f}, fired {np.isfinite(ctx['t']).mean():.3f}", flush=True)
    return mus


if __name__ == "__main__":
    import sys
    from paper_2607_14672_gb300 import configs
    which = sys.argv[1:] or ["2", "3", "4", "5"]
    if "2" in which:
        print("CFG2_MU", [round(m, 5) for m in calibrate_cfg2()])
    if "3" in which:
        print("CFG3 mu*N", [round(m, 2) for m in calibrate_cfg3()])
    if "4" in which:
        print("CFG4_MU", tuple(round(m, 5) for m in calibrate_conv(configs.config4(), batch=2)))
    if "5" in which:
        print("CFG5_MU", tuple(round(m, 5) for m in calibrate_conv(configs.config5(), batch=1)))
    if "syn9" in which:
        print("SYN9_MU", tuple(round(m, 5) for m in calibrate_conv(configs.syn_snn9(mus=(0.0,) * 9), batch=2)))
    if "syn20" in which:
        print("SYN20_MU", tuple(round(m, 5) for m in calibrate_conv(configs.syn_snn20(mus=(0.0,) * 20), batch=2)))
