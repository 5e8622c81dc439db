"""Oracle, DSTD: grid, kernel, binning, forward and analytic backward (App. B).

Test infrastructure (see the package header). Float64 throughout.

Parity status: pinned.
  * ``K_dstd``: K_DSTD(0) = 1 from both branches, K_DSTD(+-dt) = 0, limits
    between the rows of Tab. DSTD_kernels, and the defining property of
    App. B.2: v^(T_m) = v(T_m) at every grid point (checked against the
    exact potential and against RK4 integration of the ODE).
  * ``solve``: table closed forms (Tab. timing_DSTD) against bracketed
    bisection; single-spike results against the exact method; convergence
    to the exact method as M grows (App. E.1).
  * ``backward_*``: central finite differences of the float64 forward.

Readings where the paper is silent or garbled (the CUDA path takes the same ones):
  R1  candidates q = 0..M-1 on [T_q, T_{q+1}); no crossing by T_M = silent;
      so only w^_m for m = 0..M-1 can matter and the bin axis has M entries.
  R2  Eq. DSTD_kernel is applied literally for m = 0..M-1: a spike earlier
      than T_{-1} = T_0 - dt contributes nothing.
  R3  a spike exactly on T_m uses the t >= 0 branch at m (K_DSTD(0) = 1).
  R4  the second case of the general-tau s_jm in App. B.2 carries a sign
      slip in one exponent; Tab. DSTD_kernels (used here) has it right.
  R5  general (tau_v, tau_I) rows without a closed form use the bracketed
      numeric root of the interval potential; (tau, inf) uses the (inf, tau)
      rows by the symmetry of K.
  R8  in the backward, dv^/dt at the spike is floored at 1e-6 V_th / dt.
"""

import numpy as np

from . import lif

INF = np.inf


def grid(t_first, t_end, M, t_offset=0.0):
    """DSTD time points T_m = T_first + m dt - t_offset, m = 0..M (App. B.1).

    dt = (T_end - T_first) / M (App. C.1); t_offset must lie in
    (-dt/2, dt/2]. Returns (T [M+1], dt).
    """
    dt = (t_end - t_first) / M
    if not (-dt / 2 < t_offset <= dt / 2):
        raise ValueError("t_offset must lie in (-dt/2, dt/2]")
    T = t_first + np.arange(M + 1) * dt - t_offset
    return T, dt


def _rho(dt, tau):
    return 1.0 if np.isinf(tau) else np.exp(-dt / tau)


def K_dstd(t, dt, tau_v, tau_I):
    """DSTD kernel K_DSTD(t) of Tab. DSTD_kernels (branch by the sign of t).

    The caller restricts t to [-dt, dt) (Eq. DSTD_kernel); this function
    only chooses the t < 0 or t >= 0 column of the table.
    """
    t = np.asarray(t, dtype=np.float64)
    case = lif.lif_case(tau_v, tau_I)
    neg = t < 0
    with np.errstate(over="ignore", invalid="ignore"):
        if case == "inf_inf":
            left = (t + dt) / dt
            right = (dt - t) / dt
        elif case in ("inf_tau", "tau_inf"):
            tau = tau_I if case == "inf_tau" else tau_v
            r = _rho(dt, tau)
            left = (-r + np.exp(t / tau)) / (1.0 - r)
            right = (1.0 - np.exp((t - dt) / tau)) / (1.0 - r)
        elif case == "tau_tau":
            tau = tau_v
            left = (t + dt) / dt * np.exp(t / tau)
            right = (dt - t) / dt * np.exp(t / tau)
        else:  # tau_v != tau_I row; the (2 tau, tau) row is the same formula
            rv, ri = _rho(dt, tau_v), _rho(dt, tau_I)
            den = rv - ri
            left = (-ri * np.exp(t / tau_v) + rv * np.exp(t / tau_I)) / den
            right = (np.exp((t - dt) / tau_v) - np.exp((t - dt) / tau_I)) / den
    return np.where(neg, left, right)


def K_dstd_prime(t, dt, tau_v, tau_I):
    """d K_DSTD / dt, derivative of each column of Tab. DSTD_kernels.

    At t = 0 the t >= 0 column is used (one-sided, reading R3).
    """
    t = np.asarray(t, dtype=np.float64)
    case = lif.lif_case(tau_v, tau_I)
    neg = t < 0
    with np.errstate(over="ignore", invalid="ignore"):
        if case == "inf_inf":
            left = np.full_like(t, 1.0 / dt)
            right = np.full_like(t, -1.0 / dt)
        elif case in ("inf_tau", "tau_inf"):
            tau = tau_I if case == "inf_tau" else tau_v
            r = _rho(dt, tau)
            left = np.exp(t / tau) / (tau * (1.0 - r))
            right = -np.exp((t - dt) / tau) / (tau * (1.0 - r))
        elif case == "tau_tau":
            tau = tau_v
            e = np.exp(t / tau)
            left = e * (1.0 / dt + (t + dt) / (dt * tau))
            right = e * (-1.0 / dt + (dt - t) / (dt * tau))
        else:
            rv, ri = _rho(dt, tau_v), _rho(dt, tau_I)
            den = rv - ri
            left = (-ri * np.exp(t / tau_v) / tau_v + rv * np.exp(t / tau_I) / tau_I) / den
            right = (np.exp((t - dt) / tau_v) / tau_v - np.exp((t - dt) / tau_I) / tau_I) / den
    return np.where(neg, left, right)


def _extended_grid(T, dt):
    """T_{-1}, T_0, ..., T_M with T_{-1} = T_0 - dt."""
    return np.concatenate([[T[0] - dt], T])


def binning(t_in, T, dt, tau_v, tau_I, derivative=False):
    """Event weights s_jm of Eq. DSTD_kernel for m = 0..M-1 (reading R1).

    s_jm = K_DSTD(t_j - T_m) if T_{m-1} <= t_j < T_{m+1}, else 0; silent
    inputs (+inf) give no entries. t_in [..., N_in] -> s [..., M, N_in].
    With ``derivative`` the result is d s_jm / d t_j instead.
    """
    t_in = np.asarray(t_in, float)
    M = T.size - 1
    Te = _extended_grid(T, dt)          # Te[m + 1] = T_m
    tj = t_in[..., None, :]             # [..., 1, N]
    Tm = Te[1:M + 1][:, None]           # [M, 1]
    lo = Te[0:M][:, None]               # T_{m-1}
    hi = Te[2:M + 2][:, None]           # T_{m+1}
    with np.errstate(invalid="ignore"):
        inside = np.isfinite(tj) & (tj >= lo) & (tj < hi)
    d = np.where(inside, tj - Tm, 0.0)
    f = K_dstd_prime if derivative else K_dstd
    return np.where(inside, f(d, dt, tau_v, tau_I), 0.0)


def solve(what, T, dt, tau_v, tau_I, v_th, solver="table"):
    """First spike time from the discretised inputs w^ (Tab. timing_DSTD).

    what [..., N, M]: w^_im for m = 0..M-1 (the grid weights of Eq. DSTD).
    On interval q the potential is sum_{m<=q} w^_im K(t - T_m); its candidate
    t_iq comes from Tab. timing_DSTD (``solver="table"``; the general row,
    which the table lacks, and ``solver="numeric"`` use bisection), and
    t^_i = min_q { t_iq : T_q <= t_iq < T_{q+1} } (Eq. timing_DSTD).

    Returns dict:
      t      [..., N] spike times (+inf = silent)
      q      [..., N] index of the interval holding the spike (M if silent)
      vpeak  [..., N] max of v^ over [T_0, T_{q+1}] (whole window if silent)
      vdot   [..., N] dv^/dt at the spike (nan if silent), by direct sum
    """
    what = np.asarray(what, float)
    M = T.size - 1
    case = lif.lif_case(tau_v, tau_I)
    lo = T[:M]
    hi = T[1:M + 1]
    c = lif.interval_coeffs(case, tau_v, tau_I, np.broadcast_to(lo, what.shape), what, T[0])
    cand = None
    if solver == "table":
        cand = lif.closed_form_candidate(c, v_th, table="dstd")
    if cand is None:
        cand = lif.numeric_candidate(c, lo, hi, v_th)
    with np.errstate(invalid="ignore"):
        valid = np.isfinite(cand) & (cand >= lo) & (cand < hi)
    fired = valid.any(-1)
    q = np.where(fired, np.argmax(valid, -1), M)
    t = np.where(fired, np.take_along_axis(cand, np.minimum(q, M - 1)[..., None], -1)[..., 0], INF)
    peaks = lif.interval_peak(c, lo, hi)
    upto = np.arange(M) <= np.minimum(q, M - 1)[..., None]
    vpeak = np.max(np.where(upto, peaks, -np.inf), -1)
    # dv^/dt at the spike by the direct sum over grid weights (Eq. Vmem_analytical)
    ts = np.where(fired, t, T[0])[..., None]
    vdot = np.sum(np.where(upto, what * lif.K_prime(ts - lo, tau_v, tau_I), 0.0), -1)
    vdot = np.where(fired, vdot, np.nan)
    return {"t": t, "q": q, "vpeak": vpeak, "vdot": vdot, "fired": fired}


def vdot_floor(v_th, dt):
    """Reading R8: lower bound on dv^/dt at a spike used in the backward."""
    return 1e-6 * v_th / dt


def solve_backward(ctx, g_t, T, dt, tau_v, tau_I, v_th):
    """d C / d w^_im from d C / d t_i, by the implicit function theorem.

    v^(t_i) = V_th with v^(t) = sum_{m<=q} w^_m K(t - T_m) gives
    d t_i / d w^_im = -K(t_i - T_m) / v^'(t_i) for m <= q_i and 0 for later m;
    silent neurons get no gradient. Returns g_what [..., N, M].
    """
    M = T.size - 1
    fired = ctx["fired"]
    g = np.where(fired, np.asarray(g_t, float), 0.0)
    vd = np.maximum(np.where(fired, ctx["vdot"], 1.0), vdot_floor(v_th, dt))
    ts = np.where(fired, ctx["t"], T[0])[..., None]
    Km = lif.K(ts - T[:M], tau_v, tau_I)
    upto = np.arange(M) <= np.minimum(ctx["q"], M - 1)[..., None]
    return np.where(upto & fired[..., None], -g[..., None] * Km / vd[..., None], 0.0)


# ---------------------------------------------------------------------------
# Dense layer: w^_im = sum_j w_ij s_jm (Eq. DSTD).
# ---------------------------------------------------------------------------

def forward_dense(t_in, W, T, dt, tau_v, tau_I, v_th, solver="table"):
    """One DSTD layer (Alg. 2 body): binning, contraction, candidate solve.

    t_in [B, N_in], W [N_out, N_in] -> dict of ``solve`` plus s [B, M, N_in]
    and what [B, N_out, M].
    """
    s = binning(t_in, T, dt, tau_v, tau_I)
    what = np.einsum("bmj,ij->bim", s, np.asarray(W, float))
    ctx = solve(what, T, dt, tau_v, tau_I, v_th, solver)
    ctx.update(s=s, what=what)
    return ctx


def backward_dense(ctx, t_in, W, g_t, T, dt, tau_v, tau_I, v_th):
    """Gradients of one dense DSTD layer.

    g_t [B, N_out] = dC/dt_out. Returns (g_W [N_out, N_in], g_t_in [B, N_in],
    g_what [B, N_out, M]):
      g_W_ij   = sum_b sum_m g_what_bim s_bjm
      g_t_in_j = sum_m (sum_i w_ij g_what_bim) d s_bjm / d t_bj.
    """
    gw = solve_backward(ctx, g_t, T, dt, tau_v, tau_I, v_th)
    s = ctx["s"]
    g_W = np.einsum("bim,bmj->ij", gw, s)
    gS = np.einsum("bim,ij->bmj", gw, np.asarray(W, float))
    ds = binning(t_in, T, dt, tau_v, tau_I, derivative=True)
    g_t_in = np.sum(gS * ds, axis=1)
    return g_W, g_t_in, gw
