"""Pins for oracle.dstd: Tab. DSTD_kernels identities, the App. B.2 exactness
property, agreement with the exact method, convergence in M (App. E.1),
invariants, and finite-difference gradients of the analytic backward."""

import numpy as np
import pytest

from oracle import dstd, exact, lif

INF = np.inf

TAUS = [(0.5, 0.25), (0.4, 0.4), (INF, 0.3), (0.3, INF), (INF, INF), (1.0, 0.25), (0.25, 0.5)]
WMEAN = {(0.5, 0.25): 1.2, (0.4, 0.4): 0.9, (INF, 0.3): 0.4, (0.3, INF): 0.4, (INF, INF): 0.25,
         (1.0, 0.25): 0.8, (0.25, 0.5): 1.2}


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_kernel_identities(tau_v, tau_I):
    dt = 0.07
    # K_DSTD(0) = 1 from either side, K_DSTD(-dt) = 0, K_DSTD(dt^-) -> 0, K_DSTD >= 0
    assert abs(dstd.K_dstd(0.0, dt, tau_v, tau_I) - 1.0) < 1e-13
    assert abs(dstd.K_dstd(-1e-13, dt, tau_v, tau_I) - 1.0) < 1e-10
    assert abs(dstd.K_dstd(-dt, dt, tau_v, tau_I)) < 1e-13
    assert abs(dstd.K_dstd(dt * (1 - 1e-13), dt, tau_v, tau_I)) < 1e-10
    t = np.linspace(-dt, dt, 2001)[:-1]
    assert (dstd.K_dstd(t, dt, tau_v, tau_I) >= -1e-14).all()


def test_kernel_row_limits():
    dt = 0.05
    t = np.linspace(-dt, dt, 401)[:-1]
    tau = 0.3
    np.testing.assert_allclose(dstd.K_dstd(t, dt, tau * (1 + 1e-5), tau),
                               dstd.K_dstd(t, dt, tau, tau), rtol=0, atol=1e-5)
    np.testing.assert_allclose(dstd.K_dstd(t, dt, 1e8, tau), dstd.K_dstd(t, dt, INF, tau), rtol=0, atol=1e-7)
    np.testing.assert_allclose(dstd.K_dstd(t, dt, INF, 1e8), dstd.K_dstd(t, dt, INF, INF), rtol=0, atol=1e-7)
    # symmetry of the kernel under tau_v <-> tau_I carries over to K_DSTD
    np.testing.assert_allclose(dstd.K_dstd(t, dt, 0.5, 0.25), dstd.K_dstd(t, dt, 0.25, 0.5), rtol=1e-12)
    # the (2 tau, tau) row is the tau_v != tau_I row at tau_v = 2 tau_I
    np.testing.assert_allclose(dstd.K_dstd(t, dt, 0.5, 0.25), dstd.K_dstd(t, dt, 0.5 * (1 + 1e-10), 0.25),
                               rtol=1e-8, atol=1e-12)


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_kernel_derivative_by_finite_difference(tau_v, tau_I):
    dt = 0.08
    t = np.concatenate([np.linspace(-dt + 1e-4, -1e-4, 40), np.linspace(1e-4, dt - 1e-4, 40)])
    h = 1e-7
    fd = (dstd.K_dstd(t + h, dt, tau_v, tau_I) - dstd.K_dstd(t - h, dt, tau_v, tau_I)) / (2 * h)
    np.testing.assert_allclose(dstd.K_dstd_prime(t, dt, tau_v, tau_I), fd, rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
@pytest.mark.parametrize("t_offset", [0.0, 0.013])
def test_exact_at_grid_points(tau_v, tau_I, t_offset):
    # App. B.2: the discretised potential equals the exact one at every T_m,
    # checked against the analytic superposition and against RK4 of the ODE.
    M = 24
    T, dt = dstd.grid(0.0, 1.2, M, t_offset)
    g = np.random.default_rng(2)
    t_in = g.uniform(T[0], T[-1], (1, 40))
    t_in[0, :5] = INF
    w = g.normal(0.3, 1.0, (3, 40))
    ctx = dstd.forward_dense(t_in, w, T, dt, tau_v, tau_I, 1e9)   # threshold out of reach
    what = ctx["what"][0]                                          # [3, M]
    vhat = np.stack([(what[:, :min(m + 1, M)] * lif.K(T[m] - T[:min(m + 1, M)], tau_v, tau_I)).sum(1)
                     for m in range(M + 1)], 1)
    fin = np.isfinite(t_in[0])
    v = np.stack([(w[:, fin] * lif.K(T[m] - t_in[0, fin], tau_v, tau_I)).sum(1) for m in range(M + 1)], 1)
    np.testing.assert_allclose(vhat, v, rtol=0, atol=1e-12)
    v_ode = lif.ode_trajectory(t_in[0], w[0], tau_v, tau_I, T, h=2e-4)
    np.testing.assert_allclose(vhat[0], v_ode, rtol=0, atol=1e-10)


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_exact_after_next_grid_point(tau_v, tau_I):
    # one spike in [T_k, T_{k+1}): v^(t) = v(t) for every t >= T_{k+1}
    T, dt = dstd.grid(0.0, 1.0, 20)
    t0 = T[6] + 0.37 * dt
    what = dstd.forward_dense(np.array([[t0]]), np.array([[1.0]]), T, dt, tau_v, tau_I, 1e9)["what"][0, 0]
    te = np.linspace(T[7], T[-1] - 1e-9, 300)
    m_of = np.floor((te - T[0]) / dt).astype(int)
    vhat = np.array([np.sum(what[:m + 1] * lif.K(x - T[:m + 1], tau_v, tau_I)) for x, m in zip(te, m_of)])
    np.testing.assert_allclose(vhat, lif.K(te - t0, tau_v, tau_I), rtol=0, atol=1e-12)


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_single_spike_time_equals_exact(tau_v, tau_I):
    # a crossing after the grid point following the input is exact under DSTD
    T, dt = dstd.grid(0.0, 2.0, 40)
    t0 = T[3] + 0.61 * dt
    w = {(INF, INF): 2.0}.get((tau_v, tau_I), 30.0)
    ex = exact.exact_forward(np.array([[t0]]), np.array([[w]]), tau_v, tau_I, 1.0)[0, 0]
    assert ex > T[4]
    for solver in ("table", "numeric"):
        d = dstd.forward_dense(np.array([[t0]]), np.array([[w]]), T, dt, tau_v, tau_I, 1.0, solver)["t"][0, 0]
        assert abs(d - ex) < 1e-10


@pytest.mark.parametrize("tau_v,tau_I", [(0.5, 0.25), (0.4, 0.4), (INF, 0.3), (0.3, INF), (INF, INF)])
def test_table_matches_numeric(tau_v, tau_I):
    T, dt = dstd.grid(0.0, 1.2, 32, 0.011)
    g = np.random.default_rng(9)
    t_in = g.uniform(0, 1.0, (16, 48))
    t_in[g.random(t_in.shape) < 0.2] = INF
    W = g.normal(WMEAN[(tau_v, tau_I)] / 2, 0.6, (64, 48))
    a = dstd.forward_dense(t_in, W, T, dt, tau_v, tau_I, 1.0, "table")
    b = dstd.forward_dense(t_in, W, T, dt, tau_v, tau_I, 1.0, "numeric")
    ok = np.abs(a["vpeak"] - 1.0) > 1e-7
    np.testing.assert_array_equal(a["fired"][ok], b["fired"][ok])
    both = ok & a["fired"] & b["fired"]
    assert both.sum() > 100
    np.testing.assert_allclose(a["t"][both], b["t"][both], rtol=0, atol=1e-9)
    np.testing.assert_array_equal(a["q"][both], b["q"][both])


@pytest.mark.parametrize("tau_v,tau_I", [(0.4, 0.2), (INF, INF), (INF, 0.3), (1.0, 0.25)])
def test_converges_to_exact_as_M_grows(tau_v, tau_I):
    # App. E.1 / Sec. 3: the DSTD error falls as the number of steps grows
    g = np.random.default_rng(1)
    t_in = g.uniform(0, 1, (4, 200))
    W = g.normal(WMEAN.get((tau_v, tau_I), 1.2) * 12 / 200, 0.15, (40, 200))
    ex = exact.exact_forward(t_in, W, tau_v, tau_I, 1.0, t_end=2.0)
    rmse, med = {}, {}
    for M in (5, 10, 20, 40, 80, 160, 320, 640):
        T, dt = dstd.grid(0.0, 2.0, M)
        d = dstd.forward_dense(t_in, W, T, dt, tau_v, tau_I, 1.0)
        both = np.isfinite(ex) & d["fired"]
        assert both.sum() > 40
        e = np.abs(d["t"][both] - ex[both])
        rmse[M] = np.sqrt(np.mean(e ** 2))
        med[M] = np.median(e)
    assert rmse[20] < rmse[5]
    assert rmse[640] < 0.01 * rmse[5]
    assert rmse[640] < 1e-4
    # the typical error falls with every doubling of M (single near-tangent
    # neurons can jump, so the median, not the max, is checked)
    Ms = sorted(med)
    for a, b in zip(Ms, Ms[1:]):
        assert med[b] < med[a]


def test_invariants():
    T, dt = dstd.grid(0.0, 1.2, 32, -0.01)
    g = np.random.default_rng(5)
    t_in = g.uniform(0, 1, (8, 30))
    t_in[g.random(t_in.shape) < 0.3] = INF
    W = g.normal(0.6, 1.0, (20, 30))
    base = dstd.forward_dense(t_in, W, T, dt, 0.5, 0.25, 1.0)
    t = base["t"]
    # causality: a spike can never precede the grid point before the first input
    first_in = np.min(np.where(np.isfinite(t_in), t_in, INF), 1)
    assert (t >= (first_in - dt)[:, None] - 1e-12).all()
    assert (t[np.isfinite(t)] >= T[0]).all() and (t[np.isfinite(t)] < T[-1]).all()
    # monotonicity: s >= 0 and K >= 0, so raising any weight never delays a spike
    W2 = W + np.abs(g.normal(0, 0.3, W.shape))
    t2 = dstd.forward_dense(t_in, W2, T, dt, 0.5, 0.25, 1.0)["t"]
    assert (t2 <= t + 1e-12).all()
    # silent inputs contribute nothing
    W3 = W.copy()
    W3[:, ~np.isfinite(t_in).all(0)] += 0.0
    sil = ~np.isfinite(t_in[0])
    W4 = W.copy()
    W4[:, sil] = 100.0
    t4 = dstd.forward_dense(t_in[:1], W4, T, dt, 0.5, 0.25, 1.0)["t"]
    np.testing.assert_array_equal(t4, t[:1])
    # an all-silent sample is all-silent
    tz = dstd.forward_dense(np.full((1, 30), INF), W, T, dt, 0.5, 0.25, 1.0)["t"]
    assert np.isinf(tz).all()


def test_early_spikes_are_dropped():
    # reading R2: a spike before T_{-1} = T_0 - dt has no grid weight at all
    T, dt = dstd.grid(0.5, 1.5, 10)
    s = dstd.binning(np.array([[0.5 - 1.5 * dt, 0.5 - 0.5 * dt, 0.5, 1.4 + 1e-12, 1.5]]), T, dt, 0.5, 0.25)
    assert np.all(s[0, :, 0] == 0)
    assert s[0, 0, 1] > 0 and np.all(s[0, 1:, 1] == 0)
    assert s[0, 0, 2] == 1.0
    # just after T_{M-1}: nearly all weight on m = M-1 (the rest would go to T_M)
    assert s[0, -1, 3] > 0.99
    assert np.all(s[0, :, 4] == 0)


def _loss_and_grads(t_in, W, T, dt, tv, ti, c):
    ctx = dstd.forward_dense(t_in, W, T, dt, tv, ti, 1.0)
    t = ctx["t"]
    L = np.sum(np.where(ctx["fired"], c * t, 0.0))
    gW, gt, _ = dstd.backward_dense(ctx, t_in, W, np.where(ctx["fired"], c, 0.0), T, dt, tv, ti, 1.0)
    return L, gW, gt, ctx


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_backward_by_finite_differences(tau_v, tau_I):
    T, dt = dstd.grid(0.0, 1.2, 16, 0.02)
    g = np.random.default_rng(13)
    t_in = g.uniform(0, 1, (3, 10))
    t_in[0, 2] = INF
    W = g.normal(1.3 * WMEAN[(tau_v, tau_I)], 0.8, (5, 10))
    c = g.normal(1.0, 0.5, (3, 5))
    L0, gW, gt, ctx = _loss_and_grads(t_in, W, T, dt, tau_v, tau_I, c)
    assert ctx["fired"].sum() >= 5
    h = 1e-7
    fdW = np.zeros_like(W)
    for i in range(W.shape[0]):
        for j in range(W.shape[1]):
            Wp, Wm = W.copy(), W.copy()
            Wp[i, j] += h
            Wm[i, j] -= h
            fdW[i, j] = (_loss_and_grads(t_in, Wp, T, dt, tau_v, tau_I, c)[0]
                         - _loss_and_grads(t_in, Wm, T, dt, tau_v, tau_I, c)[0]) / (2 * h)
    assert np.linalg.norm(gW - fdW) <= 1e-6 * np.linalg.norm(fdW) + 1e-9
    fdt = np.zeros_like(t_in)
    for b in range(t_in.shape[0]):
        for j in range(t_in.shape[1]):
            if not np.isfinite(t_in[b, j]):
                continue
            tp, tm = t_in.copy(), t_in.copy()
            tp[b, j] += h
            tm[b, j] -= h
            fdt[b, j] = (_loss_and_grads(tp, W, T, dt, tau_v, tau_I, c)[0]
                         - _loss_and_grads(tm, W, T, dt, tau_v, tau_I, c)[0]) / (2 * h)
    assert np.linalg.norm(gt - fdt) <= 1e-6 * np.linalg.norm(fdt) + 1e-9
    assert gt[0, 2] == 0.0


def test_weight_gradient_sign():
    # v^ grows with every w_ij (s >= 0, K >= 0): d t_i / d w_ij <= 0
    T, dt = dstd.grid(0.0, 1.2, 16)
    g = np.random.default_rng(17)
    t_in = g.uniform(0, 1, (6, 12))
    W = g.normal(1.2, 0.8, (7, 12))
    ctx = dstd.forward_dense(t_in, W, T, dt, 0.5, 0.25, 1.0)
    for i in range(7):
        gsel = np.zeros((6, 7))
        gsel[:, i] = 1.0
        gW, _, _ = dstd.backward_dense(ctx, t_in, W, gsel, T, dt, 0.5, 0.25, 1.0)
        assert (gW[i] <= 1e-15).all()
