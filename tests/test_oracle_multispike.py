"""Pins of the multi-spike oracle (App. D, Eq. Vmem_multiSpikes), CPU only."""

import numpy as np
import pytest

from oracle import dstd, exact, multispike as ms

INF = np.inf
TAUS = [(0.5, 0.25), (INF, INF), (INF, 0.3), (0.3, INF), (0.4, 0.4), (1.0, 0.25)]


def _layer(seed, B, N_in, N_out, F_in, mean=1.2, lo=0.0, hi=1.0, silent=0.2):
    g = np.random.default_rng(seed)
    t = np.sort(g.uniform(lo, hi, (B, N_in, F_in)), axis=-1)
    t[g.random(t.shape) < silent] = INF
    t = np.sort(t, axis=-1)
    W = g.normal(mean, 1.0, (N_out, N_in))
    return t, W


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_exact_multispike_matches_ode_with_reset(tau_v, tau_I):
    t, W = _layer(1, 1, 6, 4, 2, mean=2.5)
    out = ms.exact_forward_ms(t, W, tau_v, tau_I, 1.0, t_end=1.5, F_out=4)
    tt = t[0].reshape(-1)
    jj = np.repeat(np.arange(6), 2)
    fin = np.isfinite(tt)
    order = np.argsort(tt[fin], kind="stable")
    n_multi = 0
    for i in range(4):
        ref = ms.ode_spikes_reset(tt[fin][order], W[i, jj[fin][order]], tau_v, tau_I, 1.0, 1.5, 4, h=2e-4)
        got = out[0, i][np.isfinite(out[0, i])]
        assert len(ref) == len(got), (i, ref, got)
        np.testing.assert_allclose(got, ref, rtol=0, atol=1e-8)
        n_multi += len(got) >= 2
    assert n_multi >= 1                      # the reset path is exercised


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_first_spike_equals_ttfs(tau_v, tau_I):
    t, W = _layer(2, 3, 12, 8, 1)
    T, dt = dstd.grid(0.0, 1.2, 12, 0.013)
    a = ms.dstd_forward_ms(t, W, T, dt, tau_v, tau_I, 1.0, F_out=3)
    b = dstd.forward_dense(t[..., 0], W, T, dt, tau_v, tau_I, 1.0, solver="numeric")
    np.testing.assert_array_equal(np.isfinite(a["t"][..., 0]), b["fired"])
    f = b["fired"]
    assert f.sum() > 5
    np.testing.assert_allclose(a["t"][..., 0][f], b["t"][f], rtol=0, atol=1e-11)
    # exact method with the same window agrees on the first spike of on-grid inputs below


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
def test_on_grid_inputs_equal_exact_multispike(tau_v, tau_I):
    # input spikes exactly on grid points: the DSTD grid weights are the exact
    # injections, so every spike (with resets) equals the exact method's
    M, t_first, t_end = 16, 0.0, 1.6
    T, dt = dstd.grid(t_first, t_end, M, 0.0)
    g = np.random.default_rng(3)
    B, N_in, N_out, F_in = 2, 10, 6, 2
    idx = np.sort(g.integers(0, M, (B, N_in, F_in)), axis=-1)
    t = T[idx]
    t[g.random(t.shape) < 0.15] = INF
    t = np.sort(t, axis=-1)
    W = g.normal(2.0, 1.0, (N_out, N_in))
    d = ms.dstd_forward_ms(t, W, T, dt, tau_v, tau_I, 1.0, F_out=5)
    e = ms.exact_forward_ms(t, W, tau_v, tau_I, 1.0, t_end=T[M], F_out=5)
    np.testing.assert_array_equal(np.isfinite(d["t"]), np.isfinite(e))
    fin = np.isfinite(e)
    assert (np.isfinite(e).sum(-1) >= 2).sum() >= 3
    np.testing.assert_allclose(d["t"][fin], e[fin], rtol=0, atol=1e-10)


@pytest.mark.parametrize("tau_v,tau_I", [(0.5, 0.25), (INF, INF), (INF, 0.3), (1.0, 0.25)])
def test_backward_by_finite_differences(tau_v, tau_I):
    t, W = _layer(4, 2, 6, 4, 2, mean=2.2)
    T, dt = dstd.grid(0.0, 1.2, 10, 0.01)
    F = 4
    ctx = ms.dstd_forward_ms(t, W, T, dt, tau_v, tau_I, 1.0, F)
    fin = np.isfinite(ctx["t"])
    assert (fin.sum(-1) >= 2).sum() >= 2
    assert ctx["margin"].min() > 1e-4
    c = np.random.default_rng(9).normal(size=ctx["t"].shape)
    gW, gt, _ = ms.dstd_backward_ms(ctx, t, W, np.where(fin, c, 0.0), T, dt, tau_v, tau_I, 1.0)

    def obj(Wx, tx):
        r = ms.dstd_forward_ms(tx, Wx, T, dt, tau_v, tau_I, 1.0, F)
        assert np.array_equal(np.isfinite(r["t"]), fin)
        return float(np.sum(np.where(fin, c * r["t"], 0.0)))

    h = 1e-7
    fdW = np.zeros_like(W)
    for idx in np.ndindex(W.shape):
        Wp, Wm = W.copy(), W.copy()
        Wp[idx] += h
        Wm[idx] -= h
        fdW[idx] = (obj(Wp, t) - obj(Wm, t)) / (2 * h)
    assert np.linalg.norm(gW - fdW) <= 1e-6 * np.linalg.norm(fdW)
    fdt = np.zeros_like(t)
    for idx in np.ndindex(t.shape):
        if not np.isfinite(t[idx]):
            continue
        tp, tm = t.copy(), t.copy()
        tp[idx] += h
        tm[idx] -= h
        fdt[idx] = (obj(W, tp) - obj(W, tm)) / (2 * h)
    gt = np.where(np.isfinite(t), gt, 0.0)
    assert np.linalg.norm(gt - fdt) <= 1e-6 * np.linalg.norm(fdt)
