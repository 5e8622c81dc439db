"""Pins for oracle.exact (Alg. 1): brute-force ODE, Eq. spike_no_leak, single spikes."""

import numpy as np
import pytest

from oracle import exact, lif

INF = np.inf

CASES = [
    (0.5, 0.25, 1.2),     # (2 tau, tau)
    (0.4, 0.4, 0.9),      # (tau, tau)
    (INF, 0.3, 0.4),      # (inf, tau)
    (0.3, INF, 0.4),      # (tau, inf)
    (INF, INF, 0.25),     # (inf, inf)
    (1.0, 0.25, 0.8),     # general (4 tau, tau)
]


@pytest.mark.parametrize("tau_v,tau_I,wmean", CASES)
def test_exact_matches_rk4_brute_force(tau_v, tau_I, wmean):
    g = np.random.default_rng(21)
    n_in, n_out = 12, 6
    t_stop = 1.6
    for b in range(2):
        t_in = g.uniform(0, 1, n_in)
        t_in[g.random(n_in) < 0.2] = INF
        W = g.normal(wmean, 0.6, (n_out, n_in))
        ref = lif.ode_first_spike(t_in, W, tau_v, tau_I, 1.0, t_stop, h=2e-4)
        for solver in ("table", "numeric"):
            got = exact.exact_forward(t_in[None], W, tau_v, tau_I, 1.0, t_end=t_stop, solver=solver)[0]
            np.testing.assert_array_equal(np.isfinite(got), np.isfinite(ref))
            fin = np.isfinite(ref)
            np.testing.assert_allclose(got[fin], ref[fin], rtol=0, atol=1e-9)
        assert np.isfinite(ref).sum() >= 2


def test_non_leaky_closed_form():
    # Eq. spike_no_leak: t_i = (V_th + sum_{S_i} w t) / sum_{S_i} w, S_i = inputs before t_i
    g = np.random.default_rng(4)
    t_in = g.uniform(0, 1, (5, 30))
    W = g.normal(0.2, 0.3, (20, 30))
    t = exact.exact_forward(t_in, W, INF, INF, 1.0)
    n_fired = 0
    for b in range(5):
        for i in range(20):
            if not np.isfinite(t[b, i]):
                continue
            S = t_in[b] <= t[b, i]
            pred = (1.0 + np.sum(W[i, S] * t_in[b, S])) / np.sum(W[i, S])
            assert abs(pred - t[b, i]) < 1e-12
            n_fired += 1
    assert n_fired > 40


@pytest.mark.parametrize("tau_v,tau_I", [(INF, INF), (INF, 0.3), (0.3, INF), (0.5, 0.25), (1.0, 0.25), (0.4, 0.4)])
def test_single_input_spike(tau_v, tau_I):
    # one input of weight w at t0: t = t0 + first root of w K(s) = V_th
    t0, w = 0.2, 9.0
    got = exact.exact_forward(np.array([[t0, INF, INF]]), np.array([[w, 3.0, -1.0]]), tau_v, tau_I, 1.0)[0, 0]
    if np.isinf(tau_v) and np.isinf(tau_I):
        ref = t0 + 1.0 / w
    elif np.isinf(tau_v) or np.isinf(tau_I):
        tau = tau_I if np.isinf(tau_v) else tau_v
        ref = t0 - tau * np.log(1.0 - 1.0 / (w * tau))
    else:
        # first root of w K(s) = 1 on the rising branch, by dense search + bisection
        s = np.linspace(1e-9, 3, 300001)
        k = w * lif.K(s, tau_v, tau_I)
        i = np.argmax(k >= 1.0)
        lo, hi = s[i - 1], s[i]
        for _ in range(100):
            mid = 0.5 * (lo + hi)
            lo, hi = (lo, mid) if w * lif.K(mid, tau_v, tau_I) >= 1 else (mid, hi)
        ref = t0 + hi
    assert abs(got - ref) < 1e-10


def test_window_truncation_and_silence():
    t_in = np.array([[0.1, 0.2, INF]])
    W = np.array([[0.5, 0.5, 10.0], [-1.0, -1.0, 5.0]])
    t = exact.exact_forward(t_in, W, INF, INF, 1.0)
    assert abs(t[0, 0] - (1.0 + 0.05 + 0.1) / 1.0) < 1e-12
    assert np.isinf(t[0, 1])
    t2 = exact.exact_forward(t_in, W, INF, INF, 1.0, t_end=1.0)
    assert np.isinf(t2[0, 0])
    allsilent = exact.exact_forward(np.full((1, 3), INF), W, INF, INF, 1.0)
    assert np.isinf(allsilent).all()


def test_candidate_footprint():
    assert exact.candidate_bytes(128, 16384, 16384) == 128 * 16384 * 16384 * 16


# ---------------------------------------------------------------------------
# exact_backward (implicit function theorem at the spike) against central
# finite differences of exact_forward, whose roots come from the closed forms
# and the bracketed solver, not from the gradient formula.
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("tau_v,tau_I", [(0.5, 0.25), (INF, INF), (1.0, 1.0), (INF, 0.5), (1.0, 0.5), (0.8, INF)])
def test_exact_backward_matches_finite_differences(tau_v, tau_I):
    rng = np.random.default_rng(11)
    B, N_in, N_out = 2, 6, 5
    s = np.linspace(1e-3, 5.0, 5001)
    kmax = lif.K(s, tau_v, tau_I).max()
    t_in = rng.uniform(0.0, 1.0, (B, N_in))
    t_in[0, 5] = INF
    W = rng.normal(3.0 / (N_in * kmax), 0.8 / (N_in * kmax), (N_out, N_in))
    fwd = lambda ti, w: exact.exact_forward(ti, w, tau_v, tau_I, 1.0)
    t = fwd(t_in, W)
    assert np.isfinite(t).sum() >= 6
    g = rng.normal(0.0, 1.0, t.shape)
    gW, gT = exact.exact_backward(t_in, W, t, g, tau_v, tau_I)
    cost = lambda tt: float(np.sum(np.where(np.isfinite(tt), g * np.where(np.isfinite(tt), tt, 0.0), 0.0)))
    h = 1e-6
    checked = 0
    for i in range(N_out):
        for j in range(N_in):
            Wp, Wm = W.copy(), W.copy()
            Wp[i, j] += h
            Wm[i, j] -= h
            tp, tm = fwd(t_in, Wp), fwd(t_in, Wm)
            if not (np.array_equal(np.isfinite(tp), np.isfinite(t)) and np.array_equal(np.isfinite(tm), np.isfinite(t))):
                continue
            fd = (cost(tp) - cost(tm)) / (2 * h)
            assert abs(fd - gW[i, j]) <= 1e-6 * (1.0 + abs(fd)), (i, j, fd, gW[i, j])
            checked += 1
    for b in range(B):
        for j in range(N_in):
            if not np.isfinite(t_in[b, j]):
                assert gT[b, j] == 0.0
                continue
            tp_in, tm_in = t_in.copy(), t_in.copy()
            tp_in[b, j] += h
            tm_in[b, j] -= h
            tp, tm = fwd(tp_in, W), fwd(tm_in, W)
            if not (np.array_equal(np.isfinite(tp), np.isfinite(t)) and np.array_equal(np.isfinite(tm), np.isfinite(t))):
                continue
            fd = (cost(tp) - cost(tm)) / (2 * h)
            assert abs(fd - gT[b, j]) <= 1e-6 * (1.0 + abs(fd)), (b, j, fd, gT[b, j])
            checked += 1
    assert checked >= 30


def test_exact_backward_zero_pattern():
    """Silent outputs carry no gradient; an input after a neuron's spike has
    no effect on it (dt_i/dw_ij = 0), and a silent input none at all."""
    t_in = np.array([[0.1, 0.2, 5.0, INF]])
    W = np.array([[2.0, 2.0, 3.0, 1.0], [-1.0, -1.0, -1.0, -1.0]])
    t = exact.exact_forward(t_in, W, INF, INF, 1.0)
    assert np.isfinite(t[0, 0]) and t[0, 0] < 5.0 and not np.isfinite(t[0, 1])
    gW, gT = exact.exact_backward(t_in, W, t, np.ones_like(t), INF, INF)
    assert np.all(gW[1] == 0.0) and gW[0, 2] == 0.0 and gW[0, 3] == 0.0
    assert gT[0, 2] == 0.0 and gT[0, 3] == 0.0
    # non-leaky closed form: v = sum_j w_j (t - t_j) = 1 -> t = (1 + sum w t_j) / sum w
    sw = 4.0
    assert abs(t[0, 0] - (1.0 + 2.0 * 0.1 + 2.0 * 0.2) / sw) < 1e-12
    assert abs(gW[0, 0] - (-(t[0, 0] - 0.1) / sw)) < 1e-12
    assert abs(gT[0, 0] - 2.0 / sw) < 1e-12
