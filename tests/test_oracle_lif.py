"""Pins for oracle.lif: the spike kernel, Lambert W_0 and the interval solvers.

Each check compares the oracle with something other than itself: RK4
integration of the LIF ODE (Eq. LIF_model_TTFS), the tau_v <-> tau_I symmetry
of Tab. kernel, limits between rows, a library Lambert W, and an independent
root-finding route.
"""

import numpy as np
import pytest

from oracle import lif

INF = np.inf

TAUS = [
    (0.5, 0.25),     # (2 tau, tau) row
    (0.4, 0.4),      # (tau, tau) row
    (INF, 0.3),      # (inf, tau) row
    (0.3, INF),      # symmetric partner, no table row
    (INF, INF),      # non-leaky row
    (1.0, 0.25),     # general (4 tau, tau), no closed form
    (0.25, 0.5),     # general with tau_I > tau_v
]


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_kernel_matches_rk4_ode(tau_v, tau_I):
    # one input spike of weight w at t0: v(t) = w K(t - t0)  (Eq. Vmem_analytical)
    t0, w = 0.1, 1.3
    te = np.linspace(0.0, 2.0, 41)
    v_ode = lif.ode_trajectory([t0], [w], tau_v, tau_I, te, h=2e-4)
    v_k = w * lif.K(te - t0, tau_v, tau_I)
    np.testing.assert_allclose(v_ode, v_k, rtol=0, atol=1e-11)


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_kernel_superposition_matches_ode(tau_v, tau_I):
    g = np.random.default_rng(3)
    t_in = g.uniform(0, 1, 9)
    w = g.normal(0.5, 1.0, 9)
    te = np.sort(g.uniform(0, 1.5, 25))
    v_ode = lif.ode_trajectory(t_in, w, tau_v, tau_I, te, h=2e-4)
    v_k = (w * lif.K(te[:, None] - t_in[None, :], tau_v, tau_I)).sum(1)
    np.testing.assert_allclose(v_ode, v_k, rtol=0, atol=1e-10)


def test_kernel_symmetry():
    s = np.linspace(-0.5, 3, 200)
    for a, b in [(0.5, 0.25), (1.0, 0.25), (0.7, 0.3), (INF, 0.3)]:
        np.testing.assert_allclose(lif.K(s, a, b), lif.K(s, b, a), rtol=1e-13, atol=1e-15)


def test_kernel_row_limits():
    s = np.linspace(0, 2, 50)
    tau = 0.3
    # general row -> (tau, tau) row; the two differ to first order in eps s / tau
    np.testing.assert_allclose(lif.K(s, tau * (1 + 1e-5), tau), lif.K(s, tau, tau), rtol=1e-4, atol=1e-9)
    # general row -> (inf, tau) row
    np.testing.assert_allclose(lif.K(s, 1e7, tau), lif.K(s, INF, tau), rtol=1e-6, atol=1e-9)
    # (inf, tau) row -> (inf, inf) row
    np.testing.assert_allclose(lif.K(s, INF, 1e7), lif.K(s, INF, INF), rtol=1e-6, atol=1e-9)
    # (2 tau, tau) row == general formula evaluated at tau_v = 2 tau_I (1+1e-9)
    np.testing.assert_allclose(lif.K(s, 0.5, 0.25), lif.K(s, 0.5 * (1 + 1e-9), 0.25), rtol=1e-7, atol=1e-12)


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_kernel_prime_by_finite_difference(tau_v, tau_I):
    s = np.linspace(0.01, 2, 60)
    h = 1e-6
    fd = (lif.K(s + h, tau_v, tau_I) - lif.K(s - h, tau_v, tau_I)) / (2 * h)
    np.testing.assert_allclose(lif.K_prime(s, tau_v, tau_I), fd, rtol=1e-7, atol=1e-8)


def test_lambert_w0_against_scipy():
    sp = pytest.importorskip("scipy.special")
    z = np.concatenate([-1 / np.e + np.logspace(-14, -1, 30), np.linspace(-0.3, 5, 60), np.logspace(0, 12, 30)])
    ref = np.real(sp.lambertw(z, 0))
    np.testing.assert_allclose(lif.lambert_w0(z), ref, rtol=1e-12, atol=3e-7)
    assert np.isnan(lif.lambert_w0(np.array([-0.5, np.nan]))).all()


def _random_events(seed, n_out, n_ev, wmean):
    g = np.random.default_rng(seed)
    times = np.sort(g.uniform(0, 1, n_ev))
    w = g.normal(wmean, 1.0, (n_out, n_ev))
    return times, w


@pytest.mark.parametrize("tau_v,tau_I,wmean", [
    (0.5, 0.25, 0.8), (0.4, 0.4, 0.9), (INF, 0.3, 0.6), (0.3, INF, 0.6), (INF, INF, 0.5)])
def test_closed_forms_match_numeric_root(tau_v, tau_I, wmean):
    times, w = _random_events(11, 400, 20, wmean)
    case = lif.lif_case(tau_v, tau_I)
    c = lif.interval_coeffs(case, tau_v, tau_I, np.broadcast_to(times, w.shape), w, times[0])
    lo = times
    hi = np.append(times[1:], 2.0)
    for table in ("exact", "dstd"):
        cf = lif.closed_form_candidate(c, 1.0, table=table)
        nu = lif.numeric_candidate(c, lo, hi, 1.0)
        with np.errstate(invalid="ignore"):
            vcf = np.isfinite(cf) & (cf >= lo) & (cf < hi)
        vnu = np.isfinite(nu) & (nu < hi)
        # first valid interval per neuron must agree, and so must the time
        f_cf = np.where(vcf.any(1), np.argmax(vcf, 1), -1)
        f_nu = np.where(vnu.any(1), np.argmax(vnu, 1), -1)
        peak = lif.interval_peak(c, lo, hi)
        # neurons whose potential grazes the threshold are ill-conditioned
        graze = (np.abs(peak - 1.0) < 1e-7).any(1)
        ok = ~graze
        assert ok.sum() > 300
        np.testing.assert_array_equal(f_cf[ok], f_nu[ok])
        both = ok & (f_cf >= 0)
        assert both.sum() > 50
        t_cf = cf[both, f_cf[both]]
        t_nu = nu[both, f_nu[both]]
        np.testing.assert_allclose(t_cf, t_nu, rtol=0, atol=1e-9)


def test_two_tau_root_forms_agree():
    # Tab. timing_DSTD writes the (2 tau, tau) root as (b - sqrt)/(V/tau),
    # Tab. spike_timing as 2a/(b + sqrt); they are the same number.
    times, w = _random_events(5, 300, 15, 0.8)
    c = lif.interval_coeffs("two_tau_tau", 0.5, 0.25, np.broadcast_to(times, w.shape), w, times[0])
    a = lif.closed_form_candidate(c, 1.0, table="exact")
    b = lif.closed_form_candidate(c, 1.0, table="dstd")
    fin = np.isfinite(a) & np.isfinite(b)
    assert fin.sum() > 100
    np.testing.assert_allclose(a[fin], b[fin], rtol=0, atol=1e-9)


def test_interval_potential_matches_direct_sum():
    g = np.random.default_rng(8)
    for tv, ti in TAUS:
        times = np.sort(g.uniform(0, 1, 12))
        w = g.normal(0.3, 1, (5, 12))
        case = lif.lif_case(tv, ti)
        c = lif.interval_coeffs(case, tv, ti, np.broadcast_to(times, w.shape), w, times[0])
        t = times + 0.37 * np.append(np.diff(times), 0.2)   # a point inside each interval
        direct = np.array([[np.sum(w[i, :k + 1] * lif.K(t[k] - times[:k + 1], tv, ti))
                            for k in range(12)] for i in range(5)])
        np.testing.assert_allclose(lif.v_interval(c, t), direct, rtol=1e-11, atol=1e-11)
        fd = (lif.v_interval(c, t + 1e-6) - lif.v_interval(c, t - 1e-6)) / 2e-6
        np.testing.assert_allclose(lif.vdot_interval(c, t), fd, rtol=1e-6, atol=1e-6)
