"""Oracle, multi-spike regime (App. D, "Extension to multi-spike regime").

Test infrastructure (see the package header). Float64 throughout.

Parity status: pinned (tests/test_oracle_multispike.py).
  * ``exact_forward_ms`` against RK4 integration of the ODE with the reset
    (``ode_spikes_reset``);
  * ``dstd_forward_ms``: with one input spike per input and one output spike
    it equals the TTFS DSTD oracle (``dstd.forward_dense``); with every
    input spike on a grid point (where the grid weights are the exact
    injections) it equals ``exact_forward_ms``;
  * ``dstd_backward_ms`` against central finite differences of the forward.

Model. A neuron may fire several times. At each spike the membrane potential
is reset to 0 and the synaptic current is kept, so after the k-th spike at
t_k (Eq. Vmem_multiSpikes)
    v(t) = I(t_k) K(t - t_k) + sum of the kernels of the inputs after t_k.
DSTD discretises every input spike on its own and sums the grid weights of
the spikes of one input (s_jm = sum_f s_jm^f), w^ = W s, and after the k-th
spike the potential on [T_m, T_{m+1}) is
    A_k K(t - t_k) + sum_{q: t_k < T_q <= t} w^_q K(t - T_q),
    A_k = sum_{q: T_q <= t_k} w^_q e^{-(t_k - T_q)/tau_I};
the (k+1)-th spike is its first threshold crossing after t_k. Spikes are
found one after another (the paper: they cannot be computed in parallel).

Readings (as for the first spike, plus): a neuron fires at most F_out times
within the window [T_0, T_M) (its later crossings are dropped); a crossing
that lands exactly on the end of an interval belongs to the next one; the
temporal and dead-neuron penalties of the TTFS model are not defined for
this regime and are not applied.
"""

import numpy as np

from . import dstd, lif

INF = np.inf


def _rates(tau_v, tau_I):
    return (0.0 if np.isinf(tau_v) else 1.0 / tau_v), (0.0 if np.isinf(tau_I) else 1.0 / tau_I)


def _v(v0, I0, s, tau_v, tau_I):
    """v(s) from the state (v0, I0) at s = 0, no input in between."""
    av, _ = _rates(tau_v, tau_I)
    return v0 * np.exp(-av * s) + I0 * lif.K(s, tau_v, tau_I)


def _vdot(v0, I0, s, tau_v, tau_I):
    av, aI = _rates(tau_v, tau_I)
    return -av * _v(v0, I0, s, tau_v, tau_I) + I0 * np.exp(-aI * s)


def first_crossing(v0, I0, L, tau_v, tau_I, v_th):
    """First s in [0, L) with v(s) = v_th from (v0, I0), v0 < v_th; None if none.

    v(s) = c1 e^{-s/tau_v} + c2 e^{-s/tau_I} (or its equal-rate / infinite
    limits) has at most one interior extremum, where dv/ds changes sign; it
    is located by bisection on the sign of dv/ds. The crossing is then
    bracketed on the rising part and bisected to ~1e-15. Also returns the
    maximum of v over [0, L] (the closest approach to v_th).
    """
    if v0 >= v_th:
        return 0.0, v0                        # reached at the end of the previous interval
    if L <= 0.0:
        return None, v0
    d0, dL = _vdot(v0, I0, 0.0, tau_v, tau_I), _vdot(v0, I0, L, tau_v, tau_I)
    ends = [0.0, L]
    ext = None
    if (d0 > 0.0) != (dL > 0.0) and d0 != 0.0 and dL != 0.0:
        lo, hi = 0.0, L
        for _ in range(200):
            mid = 0.5 * (lo + hi)
            if (_vdot(v0, I0, mid, tau_v, tau_I) > 0.0) == (d0 > 0.0):
                lo = mid
            else:
                hi = mid
            if hi - lo <= 1e-16 * max(1.0, L):
                break
        ext = 0.5 * (lo + hi)
    vmax = max(_v(v0, I0, s, tau_v, tau_I) for s in ends + ([ext] if ext is not None else []))
    # the rising stretch that can hold the first crossing
    if ext is not None and d0 > 0.0:          # interior maximum
        a, b = 0.0, ext
    elif ext is not None:                     # interior minimum: v rises after it
        a, b = ext, L
    else:                                     # monotone
        a, b = 0.0, L
    if _v(v0, I0, b, tau_v, tau_I) < v_th:
        return None, vmax
    lo, hi = a, b
    for _ in range(300):
        mid = 0.5 * (lo + hi)
        if _v(v0, I0, mid, tau_v, tau_I) >= v_th:
            hi = mid
        else:
            lo = mid
        if hi - lo <= 1e-15 * max(1.0, L):
            break
    s = hi
    if s >= L:
        return None, vmax                     # exactly at the end: the next interval's
    return s, vmax


# ---------------------------------------------------------------------------
# Exact (event-driven) multi-spike times, and the brute-force ODE check.
# ---------------------------------------------------------------------------

def exact_neuron_ms(ev_t, ev_w, tau_v, tau_I, v_th, t_end, F_out):
    """Spike times of one neuron from sorted input events (times, weights)."""
    _, aI = _rates(tau_v, tau_I)
    out = []
    if ev_t.size == 0:
        return out
    v, I = 0.0, 0.0
    for e in range(ev_t.size):
        if ev_t[e] >= t_end:
            break
        I += ev_w[e]
        a = ev_t[e]
        b = min(ev_t[e + 1] if e + 1 < ev_t.size else INF, t_end)
        while len(out) < F_out:
            s, _ = first_crossing(v, I, b - a, tau_v, tau_I, v_th)
            if s is None:
                break
            out.append(a + s)
            I = I * np.exp(-aI * s)
            v = 0.0
            a = a + s
        if len(out) >= F_out:
            break
        L = b - a
        v, I = _v(v, I, L, tau_v, tau_I), I * np.exp(-aI * L)
    return out


def exact_forward_ms(t_in, W, tau_v, tau_I, v_th, t_end, F_out):
    """Exact spike times with reset. t_in [B, N_in, F_in] (+inf padded),
    W [N_out, N_in] -> [B, N_out, F_out] ascending, +inf padded."""
    t_in = np.asarray(t_in, float)
    W = np.asarray(W, float)
    B, N_in, F_in = t_in.shape
    out = np.full((B, W.shape[0], F_out), INF)
    for b in range(B):
        tt = t_in[b].reshape(-1)
        jj = np.repeat(np.arange(N_in), F_in)
        fin = np.isfinite(tt)
        order = np.argsort(tt[fin], kind="stable")
        ev_t, ev_j = tt[fin][order], jj[fin][order]
        for i in range(W.shape[0]):
            sp = exact_neuron_ms(ev_t, W[i, ev_j], tau_v, tau_I, v_th, t_end, F_out)
            out[b, i, :len(sp)] = sp
    return out


def ode_spikes_reset(ev_t, ev_w, tau_v, tau_I, v_th, t_stop, F_out, h=1e-4):
    """Brute force: RK4 steps of the ODE (step <= h, cut at input times); a
    crossing inside a step is located by bisection on the step length, v is
    reset to 0 there and I kept. One neuron; events sorted."""
    av, aI = _rates(tau_v, tau_I)
    out = []
    if len(ev_t) == 0:
        return out
    t, v, I, k = ev_t[0], 0.0, 0.0, 0
    while t < t_stop and len(out) < F_out:
        while k < len(ev_t) and ev_t[k] <= t:
            I += ev_w[k]
            k += 1
        nxt = ev_t[k] if k < len(ev_t) else INF
        step = min(h, nxt - t, t_stop - t)
        v1, I1 = lif._rk4(v, I, step, av, aI)
        if v1 >= v_th:
            lo, hi = 0.0, step
            for _ in range(200):
                mid = 0.5 * (lo + hi)
                if lif._rk4(v, I, mid, av, aI)[0] >= v_th:
                    hi = mid
                else:
                    lo = mid
                if hi - lo <= 1e-15 * max(1.0, abs(t)):
                    break
            out.append(t + hi)
            v, I = 0.0, lif._rk4(v, I, hi, av, aI)[1]
            t = t + hi
            continue
        v, I = v1, I1
        t = t + step
    return out


# ---------------------------------------------------------------------------
# DSTD multi-spike forward and backward.
# ---------------------------------------------------------------------------

def binning_ms(t_in, T, dt, tau_v, tau_I, derivative=False):
    """s_jm = sum_f K_DSTD(t_jf - T_m) (each spike discretised on its own).
    t_in [B, N_in, F_in] -> s [B, M, N_in]; with ``derivative``, the
    per-spike derivatives [B, M, N_in, F_in] instead."""
    t_in = np.asarray(t_in, float)
    per = [dstd.binning(t_in[..., f], T, dt, tau_v, tau_I, derivative) for f in range(t_in.shape[-1])]
    return np.stack(per, -1) if derivative else np.sum(per, axis=0)


def _potential_after(what, T, t_k, A_k, t, tau_v, tau_I):
    """v^(t) after the spike at t_k (A_k = current just after it); t_k = None:
    before the first spike (Eq. Vmem_multiSpikes with the grid weights)."""
    M = T.size - 1
    v = 0.0 if t_k is None else A_k * lif.K(t - t_k, tau_v, tau_I)
    for q in range(M):
        if T[q] <= t and (t_k is None or T[q] > t_k):
            v += what[q] * lif.K(t - T[q], tau_v, tau_I)
    return float(v)


def _current_after(what, T, t_k, A_k, t, tau_I):
    """I(t) after the spike at t_k: its current decayed, plus later bins."""
    _, aI = _rates(np.inf, tau_I)
    M = T.size - 1
    I = 0.0 if t_k is None else A_k * np.exp(-aI * (t - t_k))
    for q in range(M):
        if T[q] <= t and (t_k is None or T[q] > t_k):
            I += what[q] * np.exp(-aI * (t - T[q]))
    return float(I)


def solve_neuron_ms(what, T, tau_v, tau_I, v_th, F_out):
    """Spikes of one neuron from its grid weights w^ [M] (the literal sums
    above, evaluated at each sub-interval start). Returns dict with lists
    t, q (bin), I (current at the spike) and the closest approach of the
    searched maxima to v_th (``margin``)."""
    M = T.size - 1
    ts, qs, Is = [], [], []
    margin = INF
    t_k, A_k = None, 0.0
    for m in range(M):
        a = T[m]
        while len(ts) < F_out:
            if t_k is not None and t_k > a:
                a = t_k
            v0 = _potential_after(what, T, t_k, A_k, a, tau_v, tau_I)
            I0 = _current_after(what, T, t_k, A_k, a, tau_I)
            s, vmax = first_crossing(v0, I0, T[m + 1] - a, tau_v, tau_I, v_th)
            margin = min(margin, abs(vmax - v_th))
            if s is None:
                break
            t_new = a + s
            A_new = _current_after(what, T, t_k, A_k, t_new, tau_I)
            ts.append(t_new)
            qs.append(m)
            Is.append(A_new)
            t_k, A_k = t_new, A_new
        if len(ts) >= F_out:
            break
    return {"t": ts, "q": qs, "I": Is, "margin": margin}


def dstd_forward_ms(t_in, W, T, dt, tau_v, tau_I, v_th, F_out):
    """Multi-spike DSTD layer. t_in [B, N_in, F_in] -> dict with t [B, N_out,
    F_out] (ascending, +inf padded), q, I, vdot (dv^/dt at each spike,
    -v_th/tau_v + I), margin [B, N_out], s [B, M, N_in], what [B, N_out, M]."""
    av, _ = _rates(tau_v, tau_I)
    s = binning_ms(t_in, T, dt, tau_v, tau_I)
    what = np.einsum("bmj,ij->bim", s, np.asarray(W, float))
    B, N_out, _ = what.shape
    t = np.full((B, N_out, F_out), INF)
    q = np.full((B, N_out, F_out), T.size - 1, dtype=int)
    I = np.zeros((B, N_out, F_out))
    margin = np.full((B, N_out), INF)
    for b in range(B):
        for i in range(N_out):
            r = solve_neuron_ms(what[b, i], T, tau_v, tau_I, v_th, F_out)
            n = len(r["t"])
            t[b, i, :n] = r["t"]
            q[b, i, :n] = r["q"]
            I[b, i, :n] = r["I"]
            margin[b, i] = r["margin"]
    vdot = np.where(np.isfinite(t), -av * v_th + I, np.nan)
    return {"t": t, "q": q, "I": I, "vdot": vdot, "margin": margin, "s": s, "what": what}


def solve_backward_ms(ctx, g_t, T, dt, tau_v, tau_I, v_th):
    """dC/dw^ [B, N_out, M] from dC/dt [B, N_out, F_out].

    Spike k >= 1 solves v(t_k) = v_th with
        v(t) = I_{k-1} K(t - t_{k-1}) + sum_{t_{k-1} < T_q <= t} w^_q K(t - T_q),
        I_{k-1} = sum_{T_q <= t_{k-1}} w^_q e^{-aI (t_{k-1} - T_q)},
    so by the implicit function theorem, with v'_k = -av v_th + I_k,
        dt_k/dw^_q = -[e^{-aI (t_{k-1} - T_q)} K(t_k - t_{k-1})] / v'_k   (T_q <= t_{k-1})
                   = -K(t_k - T_q) / v'_k                                 (t_{k-1} < T_q <= t_k)
        dt_k/dt_{k-1} = -I_{k-1} [(av - aI) K(s) - e^{-aI s}] / v'_k,  s = t_k - t_{k-1}
    (dI/dt = -aI I between grid points, dK/ds = -av K + e^{-aI s}); the
    first spike has the TTFS form. The adjoints run from the last spike
    back to the first.
    """
    av, aI = _rates(tau_v, tau_I)
    M = T.size - 1
    t, q, I = ctx["t"], ctx["q"], ctx["I"]
    B, N, F = t.shape
    floor = dstd.vdot_floor(v_th, dt)
    gw = np.zeros((B, N, M))
    for b in range(B):
        for i in range(N):
            n = int(np.isfinite(t[b, i]).sum())
            if n == 0:
                continue
            vd = np.maximum(-av * v_th + I[b, i, :n], floor)
            adj = np.array(g_t[b, i, :n], float)
            for k in range(n - 1, 0, -1):
                sk = t[b, i, k] - t[b, i, k - 1]
                dv_dprev = I[b, i, k - 1] * ((av - aI) * lif.K(sk, tau_v, tau_I) - np.exp(-aI * sk))
                adj[k - 1] += adj[k] * (-dv_dprev / vd[k])
            for k in range(n):
                tk = t[b, i, k]
                for m in range(M):
                    if m > q[b, i, k]:
                        break
                    if k == 0:
                        basis = lif.K(tk - T[m], tau_v, tau_I)
                    elif m <= q[b, i, k - 1]:
                        basis = np.exp(-aI * (t[b, i, k - 1] - T[m])) * lif.K(tk - t[b, i, k - 1], tau_v, tau_I)
                    else:
                        basis = lif.K(tk - T[m], tau_v, tau_I)
                    gw[b, i, m] += -adj[k] * basis / vd[k]
    return gw


def dstd_backward_ms(ctx, t_in, W, g_t, T, dt, tau_v, tau_I, v_th):
    """(g_W [N_out, N_in], g_t_in [B, N_in, F_in], g_what) of one layer."""
    gw = solve_backward_ms(ctx, g_t, T, dt, tau_v, tau_I, v_th)
    g_W = np.einsum("bim,bmj->ij", gw, ctx["s"])
    gS = np.einsum("bim,ij->bmj", gw, np.asarray(W, float))
    ds = binning_ms(t_in, T, dt, tau_v, tau_I, derivative=True)       # [B, M, N_in, F_in]
    g_t_in = np.sum(gS[..., None] * ds, axis=1)
    return g_W, g_t_in, gw
