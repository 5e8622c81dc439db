"""Oracle, neuron model: LIF spike kernel, ODE brute force, candidate solvers.

Test infrastructure (see the package header). Float64 throughout.

Parity status: pinned.
  * ``K`` against brute-force RK4 integration of Eq. LIF_model_TTFS
    (``ode_first_spike``/``ode_trajectory``), and the symmetry of K under
    tau_v <-> tau_I.
  * ``closed_form_candidate`` (Tab. spike_timing / Tab. timing_DSTD) against
    ``numeric_candidate`` (bracketed bisection, an independent route).
  * ``lambert_w0`` against ``scipy.special.lambertw``.

The LIF model (Eq. LIF_model_TTFS, App. A):
    dv/dt = -v/tau_v + I,   dI/dt = -I/tau_I + sum_j w_j delta(t - t_j),
a neuron fires once, at the first t with v(t) = V_th. Its membrane potential
is v(t) = sum_j w_j K(t - t_j) (Eq. Vmem_analytical) with K from Tab. kernel.

Between two consecutive events (input spikes for the exact method, grid
points for DSTD) v(t) is a fixed combination of exponentials whose
coefficients are prefix sums over the events seen so far; Tab. spike_timing
and Tab. timing_DSTD name these sums a and b. ``interval_coeffs`` builds
them, ``v_interval``/``vdot_interval`` evaluate v on an interval,
``closed_form_candidate`` applies the tables' candidate formulas and
``numeric_candidate`` finds the first root by bisection.
"""

import numpy as np

INF = np.inf

# Rows of Tab. kernel. "tau_inf" (tau_v finite, tau_I infinite) is not a row;
# K is symmetric under tau_v <-> tau_I, so it is the (inf, tau) row with
# tau = tau_v.
CASES = ("general", "tau_tau", "two_tau_tau", "inf_tau", "tau_inf", "inf_inf")


def lif_case(tau_v, tau_I, rtol_equal=1e-6):
    """Classify (tau_v, tau_I) into a row of Tab. kernel.

    tau_v == tau_I is recognised within a relative ``rtol_equal``; the
    (2 tau, tau) row needs tau_v == 2 tau_I to 1e-12.
    """
    iv, ii = np.isinf(tau_v), np.isinf(tau_I)
    if iv and ii:
        return "inf_inf"
    if iv:
        return "inf_tau"
    if ii:
        return "tau_inf"
    if tau_v <= 0 or tau_I <= 0:
        raise ValueError("time constants must be positive or +inf")
    if abs(tau_v - tau_I) <= rtol_equal * max(tau_v, tau_I):
        return "tau_tau"
    if abs(tau_v - 2.0 * tau_I) <= 1e-12 * tau_v:
        return "two_tau_tau"
    return "general"


def K(s, tau_v, tau_I):
    """Spike kernel K(s) of Tab. kernel: v response to one unit input at s=0.

    theta(s) is taken as 1 for s > 0 and 0 otherwise (K(0) = 0 in every row).
    """
    s = np.asarray(s, dtype=np.float64)
    case = lif_case(tau_v, tau_I)
    pos = s > 0
    sp = np.where(pos, s, 0.0)
    if case == "inf_inf":
        out = sp
    elif case == "inf_tau":
        out = tau_I * (1.0 - np.exp(-sp / tau_I))
    elif case == "tau_inf":
        out = tau_v * (1.0 - np.exp(-sp / tau_v))
    elif case == "tau_tau":
        out = sp * np.exp(-sp / tau_v)
    elif case == "two_tau_tau":
        tau = tau_I
        out = 2.0 * tau * (np.exp(-sp / (2.0 * tau)) - np.exp(-sp / tau))
    else:
        out = tau_v * tau_I / (tau_v - tau_I) * (np.exp(-sp / tau_v) - np.exp(-sp / tau_I))
    return np.where(pos, out, 0.0)


def K_prime(s, tau_v, tau_I):
    """dK/ds for s > 0 (derivative of each row of Tab. kernel); 0 for s <= 0."""
    s = np.asarray(s, dtype=np.float64)
    case = lif_case(tau_v, tau_I)
    pos = s > 0
    sp = np.where(pos, s, 0.0)
    if case == "inf_inf":
        out = np.ones_like(sp)
    elif case == "inf_tau":
        out = np.exp(-sp / tau_I)
    elif case == "tau_inf":
        out = np.exp(-sp / tau_v)
    elif case == "tau_tau":
        out = np.exp(-sp / tau_v) * (1.0 - sp / tau_v)
    elif case == "two_tau_tau":
        tau = tau_I
        out = -np.exp(-sp / (2.0 * tau)) + 2.0 * np.exp(-sp / tau)
    else:
        kap = tau_v * tau_I / (tau_v - tau_I)
        out = kap * (-np.exp(-sp / tau_v) / tau_v + np.exp(-sp / tau_I) / tau_I)
    return np.where(pos, out, 0.0)


# ---------------------------------------------------------------------------
# Brute force: RK4 integration of the ODE itself (Eq. LIF_model_TTFS).
# ---------------------------------------------------------------------------

def _rate(tau):
    return 0.0 if np.isinf(tau) else 1.0 / tau


def _rk4(v, I, h, av, aI):
    """One classical RK4 step of dv/dt = -av v + I, dI/dt = -aI I."""
    def f(v_, I_):
        return -av * v_ + I_, -aI * I_
    k1v, k1i = f(v, I)
    k2v, k2i = f(v + 0.5 * h * k1v, I + 0.5 * h * k1i)
    k3v, k3i = f(v + 0.5 * h * k2v, I + 0.5 * h * k2i)
    k4v, k4i = f(v + h * k3v, I + h * k3i)
    return (v + h / 6.0 * (k1v + 2 * k2v + 2 * k3v + k4v),
            I + h / 6.0 * (k1i + 2 * k2i + 2 * k3i + k4i))


def ode_trajectory(t_in, w, tau_v, tau_I, t_eval, h=1e-4):
    """v(t) at the sorted times ``t_eval`` for one neuron, by RK4 with step <= h.

    Input spikes (finite entries of ``t_in`` with weights ``w``) jump I by w
    at their exact times; v is continuous. No threshold (subthreshold
    trajectory), used to pin K and the DSTD interpolation property.
    """
    av, aI = _rate(tau_v), _rate(tau_I)
    t_in = np.asarray(t_in, float)
    w = np.asarray(w, float)
    fin = np.isfinite(t_in)
    order = np.argsort(t_in[fin], kind="stable")
    ev_t = t_in[fin][order]
    ev_w = w[fin][order]
    t_eval = np.asarray(t_eval, float)
    out = np.empty_like(t_eval)
    t, v, I = (min(ev_t[0], t_eval[0]) if ev_t.size else t_eval[0]), 0.0, 0.0
    k = 0
    for n, te in enumerate(t_eval):
        while True:
            nxt = ev_t[k] if k < ev_t.size else INF
            stop = min(nxt, te)
            while t < stop:
                step = min(h, stop - t)
                v, I = _rk4(v, I, step, av, aI)
                t = t + step
            t = stop
            if k < ev_t.size and nxt <= te:
                I += ev_w[k]
                k += 1
                continue
            break
        out[n] = v
    return out


def ode_first_spike(t_in, W, tau_v, tau_I, v_th, t_stop, h=1e-4):
    """First threshold crossing of each neuron, by RK4 integration.

    t_in [N_in] input spike times (+inf = silent); W [N_out, N_in].
    Integrates all N_out neurons on one time grid of step <= h (steps are
    cut at input spike times), and locates the crossing inside the step in
    which v first reaches v_th by bisection on the length of one RK4 step
    from that step's start. Returns [N_out] spike times, +inf if no crossing
    before t_stop.
    """
    av, aI = _rate(tau_v), _rate(tau_I)
    t_in = np.asarray(t_in, float)
    W = np.atleast_2d(np.asarray(W, float))
    fin = np.isfinite(t_in)
    order = np.argsort(t_in[fin], kind="stable")
    ev_t = t_in[fin][order]
    ev_w = W[:, fin][:, order]
    n_out = W.shape[0]
    v = np.zeros(n_out)
    I = np.zeros(n_out)
    spike = np.full(n_out, INF)
    if ev_t.size == 0:
        return spike
    t = ev_t[0]
    k = 0
    while t < t_stop and np.isinf(spike).any():
        while k < ev_t.size and ev_t[k] <= t:
            I = I + ev_w[:, k]
            k += 1
        nxt = ev_t[k] if k < ev_t.size else INF
        step = min(h, nxt - t, t_stop - t)
        v1, I1 = _rk4(v, I, step, av, aI)
        hit = (v1 >= v_th) & np.isinf(spike)
        for i in np.nonzero(hit)[0]:
            lo, hi = 0.0, step
            for _ in range(200):
                mid = 0.5 * (lo + hi)
                vm, _ = _rk4(v[i], I[i], mid, av, aI)
                if vm >= v_th:
                    hi = mid
                else:
                    lo = mid
                if hi - lo <= 1e-15 * max(1.0, abs(t)):
                    break
            spike[i] = t + hi
        v, I = v1, I1
        t = t + step
    return spike


# ---------------------------------------------------------------------------
# Per-interval coefficient algebra (Tab. spike_timing, Tab. timing_DSTD).
# ---------------------------------------------------------------------------

def interval_coeffs(case, tau_v, tau_I, times, weights, t_ref):
    """Prefix sums defining v on each interval, for events (times, weights).

    ``times`` [..., Q] are the event times of the intervals in order (sorted
    input spikes for the exact method, grid points T_q for DSTD) and
    ``weights`` [..., Q] their weights (w~ or w^). Times are shifted by
    ``t_ref`` (v is invariant under a common time shift; the shift keeps the
    exp(t/tau) factors of the tables small). On interval q, with u = t - t_ref:

      inf_inf     : a = sum w u_j,            b = sum w;      v = b u - a
      inf_tau     : a = sum w e^{u_j/tau_I},  b = sum w;      v = tau_I (b - a e^{-u/tau_I})
      tau_inf     : a = sum w e^{u_j/tau_v},  b = sum w;      v = tau_v (b - a e^{-u/tau_v})
      tau_tau     : a = sum w e^{u_j/tau},    b = sum w (u_j/tau) e^{u_j/tau};
                                                              v = e^{-u/tau} (u a - tau b)
      two_tau_tau : a = sum w e^{u_j/tau},    b = sum w e^{u_j/(2 tau)}  (tau = tau_I);
                                                              v = 2 tau (b e^{-u/2tau} - a e^{-u/tau})
      general     : a = sum w e^{u_j/tau_v},  b = sum w e^{u_j/tau_I};
                                                              v = kappa (a e^{-u/tau_v} - b e^{-u/tau_I}),
                    kappa = tau_v tau_I / (tau_v - tau_I).

    The sums run over the events of intervals 0..q (cumulative along the
    last axis). Returns a dict with the case, constants and arrays a, b.
    """
    u = np.asarray(times, float) - t_ref
    w = np.asarray(weights, float)
    if case == "inf_inf":
        a, b = np.cumsum(w * u, -1), np.cumsum(w, -1)
    elif case == "inf_tau":
        a, b = np.cumsum(w * np.exp(u / tau_I), -1), np.cumsum(w, -1)
    elif case == "tau_inf":
        a, b = np.cumsum(w * np.exp(u / tau_v), -1), np.cumsum(w, -1)
    elif case == "tau_tau":
        e = np.exp(u / tau_v)
        a, b = np.cumsum(w * e, -1), np.cumsum(w * (u / tau_v) * e, -1)
    elif case == "two_tau_tau":
        tau = tau_I
        a, b = np.cumsum(w * np.exp(u / tau), -1), np.cumsum(w * np.exp(u / (2 * tau)), -1)
    else:
        a, b = np.cumsum(w * np.exp(u / tau_v), -1), np.cumsum(w * np.exp(u / tau_I), -1)
    return {"case": case, "tau_v": tau_v, "tau_I": tau_I, "t_ref": t_ref, "a": a, "b": b}


def v_interval(c, t):
    """v(t) on an interval from its coefficients (see ``interval_coeffs``)."""
    case, tv, ti = c["case"], c["tau_v"], c["tau_I"]
    a, b = c["a"], c["b"]
    u = np.asarray(t, float) - c["t_ref"]
    with np.errstate(over="ignore", invalid="ignore"):
        if case == "inf_inf":
            return b * u - a
        if case == "inf_tau":
            return ti * (b - a * np.exp(-u / ti))
        if case == "tau_inf":
            return tv * (b - a * np.exp(-u / tv))
        if case == "tau_tau":
            return np.exp(-u / tv) * (u * a - tv * b)
        if case == "two_tau_tau":
            tau = ti
            return 2 * tau * (b * np.exp(-u / (2 * tau)) - a * np.exp(-u / tau))
        kap = tv * ti / (tv - ti)
        return kap * (a * np.exp(-u / tv) - b * np.exp(-u / ti))


def vdot_interval(c, t):
    """dv/dt on an interval from its coefficients."""
    case, tv, ti = c["case"], c["tau_v"], c["tau_I"]
    a, b = c["a"], c["b"]
    u = np.asarray(t, float) - c["t_ref"]
    with np.errstate(over="ignore", invalid="ignore"):
        if case == "inf_inf":
            return b + 0.0 * u
        if case == "inf_tau":
            return a * np.exp(-u / ti)
        if case == "tau_inf":
            return a * np.exp(-u / tv)
        if case == "tau_tau":
            return np.exp(-u / tv) * (a - (u * a - tv * b) / tv)
        if case == "two_tau_tau":
            tau = ti
            return -b * np.exp(-u / (2 * tau)) + 2 * a * np.exp(-u / tau)
        kap = tv * ti / (tv - ti)
        return kap * (-a / tv * np.exp(-u / tv) + b / ti * np.exp(-u / ti))


def critical_time(c):
    """Time of the interior extremum of v on an interval (nan if v is monotone).

    For the two-exponential rows, dv/dt = 0 has at most one solution; the
    (inf, .) rows are monotone between events.
    """
    case, tv, ti = c["case"], c["tau_v"], c["tau_I"]
    a, b = c["a"], c["b"]
    with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
        if case in ("inf_inf", "inf_tau", "tau_inf"):
            return np.full(np.shape(a), np.nan)
        if case == "tau_tau":
            u = tv + tv * b / a
        elif case == "two_tau_tau":
            tau = ti
            # -b e^{-u/2tau} + 2 a e^{-u/tau} = 0  ->  e^{-u/2tau} = b / (2a)
            u = -2 * tau * np.log(b / (2 * a))
        else:
            # a/tv e^{-u/tv} = b/ti e^{-u/ti}  ->  u (1/ti - 1/tv) = ln(b tv / (a ti))
            u = np.log(b * tv / (a * ti)) / (1.0 / ti - 1.0 / tv)
        return np.where(np.isfinite(u), u + c["t_ref"], np.nan)


def lambert_w0(z, iters=60):
    """Principal branch W_0 of the Lambert W function, by Halley's iteration.

    Solves w e^w = z for real z >= -1/e; nan for z < -1/e (no real root) and
    for non-finite z. Starting values: the branch-point series in
    p = sqrt(2(e z + 1)) near z = -1/e, log1p(z) for moderate z and
    ln z - ln ln z for large z.
    """
    z = np.asarray(z, dtype=np.float64)
    zc = np.where(np.isfinite(z), z, 0.0)
    ok = np.isfinite(z) & (zc >= -1.0 / np.e - 1e-15)
    zc = np.where(ok, np.maximum(zc, -1.0 / np.e), 0.0)
    p = np.sqrt(np.maximum(2.0 * (np.e * zc + 1.0), 0.0))
    w_branch = -1.0 + p - p * p / 3.0 + 11.0 / 72.0 * p ** 3
    with np.errstate(divide="ignore", invalid="ignore"):
        L1 = np.log(np.maximum(zc, 1e-300))
        L2 = np.log(np.maximum(L1, 1e-300))
        w_large = L1 - L2 + L2 / np.maximum(L1, 1e-300)
    w = np.where(zc < -0.25, w_branch, np.where(zc < 3.0, np.log1p(np.maximum(zc, -0.25)), w_large))
    for _ in range(iters):
        ew = np.exp(w)
        f = w * ew - zc
        denom = ew * (w + 1.0) - (w + 2.0) * f / (2.0 * w + 2.0)
        with np.errstate(divide="ignore", invalid="ignore"):
            step = np.where((denom != 0) & np.isfinite(denom), f / denom, 0.0)
        w = np.maximum(w - np.where(np.isfinite(step), step, 0.0), -1.0)
    return np.where(ok, w, np.nan)


def closed_form_candidate(c, v_th, table="dstd"):
    """Candidate firing time of each interval from the tables' closed forms.

    ``table`` = "exact" uses Tab. spike_timing, "dstd" Tab. timing_DSTD; the
    two differ only in how the (2 tau, tau) root is written. Only the four
    tabulated rows have closed forms; (tau, inf) uses the (inf, tau) row by
    the symmetry of K. The general row has none (returns None). Invalid
    arithmetic (no real root) gives nan; validity against the interval is
    checked by the caller (Eqs. timing_exact / timing_DSTD).
    """
    case, tv, ti = c["case"], c["tau_v"], c["tau_I"]
    a, b = c["a"], c["b"]
    V = v_th
    with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
        if case == "inf_inf":
            u = (V + a) / b
        elif case in ("inf_tau", "tau_inf"):
            tau = ti if case == "inf_tau" else tv
            u = tau * np.log(a / (b - V / tau))
        elif case == "tau_tau":
            tau = tv
            z = -(V / tau) / a * np.exp(b / a)
            u = tau * (b / a - lambert_w0(z))
        elif case == "two_tau_tau":
            tau = ti
            disc = np.sqrt(b * b - 2.0 * a * V / tau)
            if table == "exact":
                u = 2 * tau * np.log(2 * a / (b + disc))
            else:
                u = 2 * tau * np.log((b - disc) / (V / tau))
        else:
            return None
    return u + c["t_ref"]


def numeric_candidate(c, lo, hi, v_th, iters=200):
    """First time in [lo, hi] with v = v_th on each interval, by bisection.

    A bracket [lo, x] with v(lo) < v_th <= v(x) is taken with x = hi if
    v(hi) >= v_th, else x = the interior extremum if v reaches v_th there.
    v on an interval has at most one extremum, so the bracket holds exactly
    one crossing. If v(lo) >= v_th already the candidate is lo. For hi = inf
    a finite right end is found by doubling. Returns nan where v stays below
    v_th on [lo, hi].
    """
    lo = np.broadcast_to(np.asarray(lo, float), np.shape(c["a"])).copy()
    hi = np.broadcast_to(np.asarray(hi, float), np.shape(c["a"])).copy()
    f = lambda t: v_interval(c, t) - v_th  # noqa: E731
    # finite right end for open last intervals
    inf_hi = np.isinf(hi)
    if inf_hi.any():
        span = np.ones_like(lo)
        hi_f = np.where(inf_hi, lo + span, hi)
        for _ in range(60):
            need = inf_hi & ~(f(hi_f) >= 0)
            if not need.any():
                break
            span = np.where(need, span * 2.0, span)
            hi_f = np.where(need, lo + span, hi_f)
        hi = hi_f
    f_lo = f(lo)
    f_hi = f(hi)
    tc = critical_time(c)
    tc_in = np.isfinite(tc) & (tc > lo) & (tc < hi)
    f_tc = np.where(tc_in, f(np.where(tc_in, tc, lo)), -np.inf)
    at_lo = f_lo >= 0
    use_hi = ~at_lo & (f_hi >= 0)
    use_tc = ~at_lo & ~use_hi & (f_tc >= 0)
    found = at_lo | use_hi | use_tc
    left = lo.copy()
    right = np.where(use_hi, hi, np.where(use_tc, tc, lo))
    active = use_hi | use_tc
    for _ in range(iters):
        mid = 0.5 * (left + right)
        fm = f(mid)
        up = fm >= 0
        right = np.where(active & up, mid, right)
        left = np.where(active & ~up, mid, left)
    cand = np.where(at_lo, lo, right)
    return np.where(found, cand, np.nan)


def interval_peak(c, lo, hi):
    """max of v over [lo, hi] on each interval (endpoints and extremum)."""
    lo = np.asarray(lo, float)
    hi = np.asarray(hi, float)
    m = np.maximum(v_interval(c, lo), v_interval(c, hi))
    tc = critical_time(c)
    tc_in = np.isfinite(tc) & (tc > lo) & (tc < hi)
    vt = np.where(tc_in, v_interval(c, np.where(tc_in, tc, lo)), -np.inf)
    return np.maximum(m, vt)
