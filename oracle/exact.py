"""Oracle, exact method: event-driven TTFS spike times (Alg. 1, App. A).

Test infrastructure (see the package header). Float64 throughout.

Parity status: pinned. Against brute-force RK4 integration of the LIF ODE on
tiny layers (``lif.ode_first_spike``), against the non-leaky closed form
Eq. spike_no_leak, and the table closed forms against the bracketed numeric
solver. ``exact_backward`` against central finite differences of
``exact_forward`` (weights and input times), and its zero pattern (silent
outputs, inputs after the spike).

Steps (Alg. 1, one layer, one sample):
  1. drop silent inputs and sort the rest, t~_1 <= ... <= t~_K;
  2. permute the weights the same way, w~_ij;
  3. on each interval [t~_k, t~_{k+1}) (t~_{K+1} = +inf) the potential is
     sum_{j<=k} w~_ij K(t - t~_j); its candidate root t_ik comes from
     Tab. spike_timing (or the numeric solver where no row applies);
  4. t_i = min_k { t_ik : t~_k <= t_ik < t~_{k+1} } (Eq. timing_exact),
     +inf if no interval holds its candidate.
An optional window end ``t_end`` closes every interval at t_end (a neuron
that has not fired by t_end is silent), which is how the exact result is
compared with DSTD on a finite window.
"""

import numpy as np

from . import lif

INF = np.inf


def exact_forward(t_in, W, tau_v, tau_I, v_th, t_end=INF, solver="table", chunk=512):
    """Exact first-spike times of one layer for a batch.

    t_in   [B, N_in]   presynaptic spike times, +inf = silent.
    W      [N_out, N_in] weights w_ij.
    solver "table" uses Tab. spike_timing where a row applies (numeric
           otherwise); "numeric" always uses bracketed bisection.
    Returns t_out [B, N_out] (+inf = silent).
    """
    t_in = np.atleast_2d(np.asarray(t_in, float))
    W = np.atleast_2d(np.asarray(W, float))
    case = lif.lif_case(tau_v, tau_I)
    B = t_in.shape[0]
    n_out = W.shape[0]
    out = np.full((B, n_out), INF)
    for b in range(B):
        fin = np.isfinite(t_in[b])
        if not fin.any():
            continue
        order = np.argsort(t_in[b][fin], kind="stable")
        tt = t_in[b][fin][order]                      # step 1: sorted times
        Wt = W[:, fin][:, order]                      # step 2: permuted weights
        lo = tt
        hi = np.minimum(np.append(tt[1:], INF), t_end)
        t_ref = tt[0]
        for i0 in range(0, n_out, chunk):
            Wc = Wt[i0:i0 + chunk]
            c = lif.interval_coeffs(case, tau_v, tau_I, np.broadcast_to(tt, Wc.shape), Wc, t_ref)
            cand = None
            if solver == "table":
                cand = lif.closed_form_candidate(c, v_th, table="exact")
            if cand is None:
                cand = lif.numeric_candidate(c, lo, hi, v_th)
            with np.errstate(invalid="ignore"):
                valid = np.isfinite(cand) & (cand >= lo) & (cand < hi) & (lo < hi)
            anyv = valid.any(-1)
            first = np.argmax(valid, -1)
            tsel = np.take_along_axis(cand, first[:, None], -1)[:, 0]
            out[b, i0:i0 + chunk] = np.where(anyv, tsel, INF)
    return out


def exact_backward(t_in, W, t_out, g_out, tau_v, tau_I):
    """Gradients through the exact spike times (the implicit function theorem
    on v_i(t_i) = v_th, Eq. Vmem_analytical at the root of Eq. timing_exact).

    Neuron i fires at t_i with v_i(t_i) = sum_j w_ij K(t_i - t_j) = v_th over
    its causal inputs (t_j < t_i: the intervals of Alg. 1 up to the one that
    holds t_i). With the slope at the crossing V'_i = sum_j w_ij K'(t_i - t_j):
        dt_i/dw_ij = -K(t_i - t_j) / V'_i,    dt_i/dt_j = w_ij K'(t_i - t_j) / V'_i.
    Silent outputs and inputs at or after t_i contribute nothing.

    t_in [B, N_in], W [N_out, N_in], t_out [B, N_out], g_out = dC/dt_out [B, N_out].
    Returns (g_W [N_out, N_in], g_t_in [B, N_in]).
    """
    t_in = np.atleast_2d(np.asarray(t_in, float))
    W = np.atleast_2d(np.asarray(W, float))
    t_out = np.atleast_2d(np.asarray(t_out, float))
    g_out = np.atleast_2d(np.asarray(g_out, float))
    fired = np.isfinite(t_out)
    x = np.where(fired[:, :, None], t_out[:, :, None], 0.0) - np.where(np.isfinite(t_in), t_in, INF)[:, None, :]
    causal = fired[:, :, None] & np.isfinite(t_in)[:, None, :] & (x > 0)
    xs = np.where(causal, x, 0.0)
    Kx = np.where(causal, lif.K(xs, tau_v, tau_I), 0.0)          # [B, N_out, N_in]
    dK = np.where(causal, lif.K_prime(xs, tau_v, tau_I), 0.0)
    Vp = np.einsum("bij,ij->bi", dK, W)                            # slope at each spike
    with np.errstate(divide="ignore", invalid="ignore"):
        dt_dv = np.where(fired, g_out / Vp, 0.0)                   # dC/dt_i / V'_i
    g_W = -np.einsum("bi,bij->ij", dt_dv, Kx)
    g_t_in = np.einsum("bi,ij,bij->bj", dt_dv, W, dK)
    return g_W, g_t_in


def candidate_bytes(B, n_in, n_out, bytes_per_candidate=16):
    """Analytic activation footprint of the exact method's candidates.

    Tab. computational_complexity: the exact formulation retains O(N_out N_in)
    candidate-dependent values per sample for reverse-mode differentiation.
    With the permuted weight, a, b and the candidate time kept per
    (sample, neuron, interval) in fp32 that is 16 bytes per candidate.
    """
    return int(B) * int(n_in) * int(n_out) * int(bytes_per_candidate)
