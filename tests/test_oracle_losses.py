"""Pins for oracle.losses and oracle.network: finite differences, AdamW against
torch.optim.AdamW, the warm-up closed form, conv == expanded dense layer, and
whole-network gradients of Eq. cost_function."""

import numpy as np
import pytest

from oracle import dstd, losses, network

INF = np.inf


def test_ce_gradient_by_finite_differences():
    g = np.random.default_rng(0)
    t = g.uniform(0.5, 1.5, (6, 10))
    t[0, 3] = INF
    lab = g.integers(0, 10, 6)
    lab[0] = 3                      # a silent target: finite loss by reading R7
    L, gr = losses.ce_loss(t, lab, 0.05, t_silent=2.0)
    assert np.isfinite(L)
    h = 1e-6
    fd = np.zeros_like(t)
    for idx in np.ndindex(t.shape):
        if not np.isfinite(t[idx]):
            continue
        tp, tm = t.copy(), t.copy()
        tp[idx] += h
        tm[idx] -= h
        fd[idx] = (losses.ce_loss(tp, lab, 0.05, 2.0)[0] - losses.ce_loss(tm, lab, 0.05, 2.0)[0]) / (2 * h)
    np.testing.assert_allclose(gr, fd, rtol=1e-6, atol=1e-8)
    assert gr[0, 3] == 0.0


def test_ce_matches_softmax_definition():
    t = np.array([[0.3, 0.5, 0.9]])
    L, _ = losses.ce_loss(t, np.array([1]), 0.1, 5.0)
    z = np.exp(-t[0] / 0.1)
    assert abs(L - (-np.log(z[1] / z.sum()))) < 1e-13


def test_temporal_penalty_value_and_gradient():
    t = np.array([[0.05, 0.5, 1.3, INF], [0.31, 0.29, 0.9, 1.0]])
    v, gr = losses.temporal_penalty(t, 0.3, 1.0, 0.05, 0.01, 0.5)
    ref = 0.5 * (0.05 * (0.05 - 0.3) ** 2 + 0.01 * (1.3 - 1.0) ** 2 + 0.05 * (0.29 - 0.3) ** 2)
    assert abs(v - ref) < 1e-15
    h = 1e-7
    for idx in np.ndindex(t.shape):
        if not np.isfinite(t[idx]):
            assert gr[idx] == 0.0
            continue
        tp, tm = t.copy(), t.copy()
        tp[idx] += h
        tm[idx] -= h
        fd = (losses.temporal_penalty(tp, 0.3, 1.0, 0.05, 0.01, 0.5)[0]
              - losses.temporal_penalty(tm, 0.3, 1.0, 0.05, 0.01, 0.5)[0]) / (2 * h)
        assert abs(fd - gr[idx]) < 1e-7


def test_dead_neuron_penalty():
    t = np.array([[INF, 0.2, INF], [INF, INF, 0.4]])
    W = np.array([[1.0, 2.0], [-1.0, 0.5], [3.0, 3.0]])
    v, cnt = losses.dead_neuron_penalty(t, W.sum(1), 0.1, 0.5)
    # Q = -sum over silent (sample, neuron) of the neuron's weight sum
    assert abs(v - (-0.1 * 0.5 * (2 * 3.0 + 1 * (-0.5) + 1 * 6.0))) < 1e-15
    np.testing.assert_array_equal(cnt, [2, 1, 1])


def test_adamw_matches_torch():
    torch = pytest.importorskip("torch")
    g = np.random.default_rng(1)
    w0 = g.normal(size=(5, 7))
    w = torch.tensor(w0.copy(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([w], lr=3e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.02)
    wn, m, v = w0.copy(), np.zeros_like(w0), np.zeros_like(w0)
    for step in range(1, 4):
        grad = g.normal(size=w0.shape)
        w.grad = torch.tensor(grad)
        opt.step()
        wn, m, v = losses.adamw_step(wn, grad, m, v, step, 3e-3, 0.9, 0.999, 1e-8, 0.02)
    np.testing.assert_allclose(wn, w.detach().numpy(), rtol=1e-12, atol=1e-14)


def test_warmup_schedule():
    for nw in range(5):
        for p in range(8):
            assert losses.warmup_lr(p, 1e-3, nw) == pytest.approx(1e-3 * 2.0 ** (min(p, nw) - nw))


def test_window_params():
    w = losses.window_params(3, 0.1, 1.0, 0.1, 0.2, 0.2)
    assert w["t_first"] == pytest.approx(0.2) and w["t_end"] == pytest.approx(1.4)
    assert w["t_head_l"] == pytest.approx(0.5) and w["t_tail_l"] == pytest.approx(1.1)


def _conv_as_dense(Wc, C, H, Wd, stride, pad):
    """Expand a conv filter into the dense matrix of the same linear map."""
    O, _, k, _ = Wc.shape
    Ho, Wo = network.conv_out_hw(H, Wd, k, stride, pad)
    D = np.zeros((O * Ho * Wo, C * H * Wd))
    for o in range(O):
        for y in range(Ho):
            for x in range(Wo):
                r = (o * Ho + y) * Wo + x
                for c in range(C):
                    for kh in range(k):
                        for kw in range(k):
                            yy, xx = y * stride + kh - pad, x * stride + kw - pad
                            if 0 <= yy < H and 0 <= xx < Wd:
                                D[r, (c * H + yy) * Wd + xx] += Wc[o, c, kh, kw]
    return D


@pytest.mark.parametrize("stride,pad,k", [(1, 1, 3), (2, 1, 3), (1, 0, 3), (1, 2, 5)])
def test_conv_equals_expanded_dense(stride, pad, k):
    g = np.random.default_rng(3)
    B, C, H, Wd, O = 2, 3, 6, 5, 4
    t_in = g.uniform(0, 1, (B, C, H, Wd))
    t_in[g.random(t_in.shape) < 0.2] = INF
    Wc = g.normal(1.0, 1.0, (O, C, k, k))
    L = dict(kind="conv", W=Wc, tau_v=0.5, tau_I=0.25, v_th=1.0, t_first=0.0, t_end=1.2, M=16,
             t_offset=0.01, stride=stride, pad=pad)
    ctx = network.forward_layer(t_in, L)
    D = _conv_as_dense(Wc, C, H, Wd, stride, pad)
    T, dt = dstd.grid(0.0, 1.2, 16, 0.01)
    ref = dstd.forward_dense(t_in.reshape(B, -1), D, T, dt, 0.5, 0.25, 1.0)
    np.testing.assert_array_equal(np.isfinite(ctx["t"].reshape(B, -1)), ref["fired"])
    fin = ref["fired"]
    np.testing.assert_allclose(ctx["t"].reshape(B, -1)[fin], ref["t"][fin], rtol=0, atol=1e-12)
    assert np.isfinite(ref["t"]).sum() > 10
    # gradients too: dW of the conv = expanded-dense dW folded back
    gt = np.where(ref["fired"], g.normal(size=ref["t"].shape), 0.0)
    gWc, gin = network.backward_layer(ctx, L, gt.reshape(ctx["t"].shape))
    gD, gin_d, _ = dstd.backward_dense(ref, t_in.reshape(B, -1), D, gt, T, dt, 0.5, 0.25, 1.0)
    np.testing.assert_allclose(gin.reshape(B, -1), gin_d, rtol=1e-10, atol=1e-12)
    # fold: dC/dWc[o,c,kh,kw] = sum of dC/dD over the entries that hold it
    fold = np.zeros_like(Wc)
    for o in range(O):
        for c in range(C):
            for kh in range(k):
                for kw in range(k):
                    e = np.zeros_like(Wc)
                    e[o, c, kh, kw] = 1.0
                    fold[o, c, kh, kw] = np.sum(gD * _conv_as_dense(e, C, H, Wd, stride, pad))
    np.testing.assert_allclose(gWc, fold, rtol=1e-10, atol=1e-12)


def _small_net(seed):
    g = np.random.default_rng(seed)
    layers = []
    sizes = [12, 9, 7, 4]
    for l in range(1, 4):
        wp = losses.window_params(l, 0.1, 1.0, 0.1, 0.2, 0.2)
        layers.append(dict(kind="dense", W=g.normal(1.8, 0.8, (sizes[l], sizes[l - 1])),
                           tau_v=0.5, tau_I=0.25, v_th=1.0, t_first=wp["t_first"], t_end=wp["t_end"],
                           M=12, t_offset=0.013 * (-1) ** l, t_head_l=wp["t_head_l"], t_tail_l=wp["t_tail_l"],
                           gamma_head=0.05, gamma_tail=0.01, gamma_q=1e-2))
    t0 = g.uniform(0, 1, (3, 12))
    t0[g.random(t0.shape) < 0.2] = INF
    return t0, layers, g.integers(0, 4, 3)


def test_network_gradients_by_finite_differences():
    t0, layers, lab = _small_net(10)
    C, parts, grads, ctxs = network.train_objective(t0, layers, lab, 0.05)
    assert all(np.isfinite(c["t"]).sum() >= 3 for c in ctxs)
    assert parts["T"] > 0 and parts["Q"] < 0
    h = 1e-7
    for l, L in enumerate(layers):
        fd = np.zeros_like(L["W"])
        for idx in np.ndindex(L["W"].shape):
            Wp, Wm = L["W"].copy(), L["W"].copy()
            Wp[idx] += h
            Wm[idx] -= h
            lp = [dict(x) for x in layers]
            lm = [dict(x) for x in layers]
            lp[l]["W"], lm[l]["W"] = Wp, Wm
            fd[idx] = (network.train_objective(t0, lp, lab, 0.05, backward=False)[0]
                       - network.train_objective(t0, lm, lab, 0.05, backward=False)[0]) / (2 * h)
        assert np.linalg.norm(grads[l] - fd) <= 1e-6 * np.linalg.norm(fd) + 1e-10, l


def _skip_net(seed, B=2):
    """conv 2->3 (3x3) - conv 3->3 (5x5, pad 2) - conv 6->4 (3x3, stride 2) whose
    input is layer 1's output delayed by 0.2 beside layer 2's (App. C.3) -
    dense readout; synfire windows as in App. C.1."""
    g = np.random.default_rng(seed)
    C0, H = 2, 5
    specs = [(3, C0, 3, 1, 1, None), (3, 3, 5, 1, 2, None), (4, 6, 3, 2, 1, (0, 0.2))]
    layers = []
    for l, (O, C, k, st, pad, skip) in enumerate(specs, start=1):
        wp = losses.window_params(l, 0.1, 1.0, 0.1, 0.2, 0.2)
        L = dict(kind="conv", W=g.normal(0.9, 0.5, (O, C, k, k)), tau_v=0.5, tau_I=0.25, v_th=1.0,
                 t_first=wp["t_first"], t_end=wp["t_end"], M=10, t_offset=0.011 * (-1) ** l, stride=st, pad=pad,
                 t_head_l=wp["t_head_l"], t_tail_l=wp["t_tail_l"], gamma_head=0.05, gamma_tail=0.01, gamma_q=1e-2)
        if skip is not None:
            L["skip"] = skip
        layers.append(L)
    wp = losses.window_params(4, 0.1, 1.0, 0.1, 0.2, 0.2)
    layers.append(dict(kind="dense", W=g.normal(0.5, 0.5, (3, 4 * 3 * 3)), tau_v=0.5, tau_I=0.25, v_th=1.0,
                       t_first=wp["t_first"], t_end=wp["t_end"], M=10, t_offset=0.0, t_head_l=wp["t_head_l"],
                       t_tail_l=wp["t_tail_l"], gamma_head=0.05, gamma_tail=0.01, gamma_q=1e-2))
    t0 = g.uniform(0, 1, (B, C0, H, H))
    t0[g.random(t0.shape) < 0.2] = INF
    return t0, layers, g.integers(0, 3, B)


def test_skip_input_is_delayed_source_then_previous():
    # the skip layer's w^ must be the sum of two separate contractions: the
    # first C_a filter channels over layer 1's spikes 0.2 later, the rest over
    # layer 2's spikes (a swapped order or a delay of the wrong sign differs)
    t0, layers, _ = _skip_net(21)
    ctxs = network.forward_net(t0, layers)
    L = layers[2]
    T, dt = network.layer_grid(L)
    B = t0.shape[0]

    def bins(t):
        return dstd.binning(t.reshape(B, -1), T, dt, L["tau_v"], L["tau_I"]).reshape((B, L["M"]) + t.shape[1:])

    a, b = ctxs[0]["t"] + 0.2, ctxs[1]["t"]
    assert np.isfinite(a).sum() > 10 and np.isfinite(b).sum() > 10
    Ca = a.shape[1]
    what = (network.conv_what(bins(a), L["W"][:, :Ca], 2, 1) + network.conv_what(bins(b), L["W"][:, Ca:], 2, 1))
    np.testing.assert_allclose(ctxs[2]["what"], what, rtol=1e-12, atol=1e-12)
    ref = dstd.solve(what.reshape(B, -1, L["M"]), T, dt, L["tau_v"], L["tau_I"], 1.0)
    t2 = ctxs[2]["t"].reshape(B, -1)
    np.testing.assert_array_equal(np.isfinite(t2), np.isfinite(ref["t"]))
    fin = np.isfinite(t2)
    assert fin.sum() > 5
    np.testing.assert_allclose(t2[fin], ref["t"][fin], rtol=0, atol=1e-12)


def test_skip_network_gradients_by_finite_differences():
    t0, layers, lab = _skip_net(22)
    C, parts, grads, ctxs = network.train_objective(t0, layers, lab, 0.05)
    assert all(np.isfinite(c["t"]).sum() >= 3 for c in ctxs)
    h = 1e-7
    g = np.random.default_rng(5)
    for l, L in enumerate(layers):
        # 12 sampled weights per layer (the whole gradient would take long)
        flat = [tuple(int(v) for v in np.unravel_index(i, L["W"].shape))
                for i in g.choice(L["W"].size, 12, replace=False)]
        for idx in flat:
            Wp, Wm = L["W"].copy(), L["W"].copy()
            Wp[idx] += h
            Wm[idx] -= h
            lp = [dict(x) for x in layers]
            lm = [dict(x) for x in layers]
            lp[l]["W"], lm[l]["W"] = Wp, Wm
            fd = (network.train_objective(t0, lp, lab, 0.05, backward=False)[0]
                  - network.train_objective(t0, lm, lab, 0.05, backward=False)[0]) / (2 * h)
            assert abs(grads[l][idx] - fd) <= 1e-6 * max(1.0, abs(fd)), (l, idx, grads[l][idx], fd)
    # the skip gradient reaches layer 1 twice (through layer 2 and the skip):
    # dropping the skip's part changes layer 1's gradient
    assert np.linalg.norm(grads[0]) > 0


def test_e_rmse():
    e, mism = network.e_rmse(np.array([1.0, 2.0, INF, 3.0]), np.array([1.1, 1.8, 1.0, 3.0]))
    assert mism == 1 and abs(e - np.sqrt((0.01 + 0.04 + 0) / 3)) < 1e-15
