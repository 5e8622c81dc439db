"""Oracle, networks: multi-layer dense / conv DSTD forward and backward.

Test infrastructure (see the package header). Float64 throughout.

Parity status: pinned. A conv layer equals a dense layer whose weight matrix
is the explicitly expanded (Toeplitz) filter; whole-network gradients against
central finite differences of ``train_objective``.

Alg. 2 (TTFS-SNN with DSTD): for l = 1..L, bin t^(l-1) on layer l's grid
(with its own t_offset), contract with W^(l) and solve for t^(l). The
objective is Eq. cost_function (``losses``); the backward runs the layers in
reverse, each adding its temporal-penalty gradient to the upstream dC/dt and
the dead-neuron term to dC/dW.

Layer spec (dict): kind ("dense" | "conv"), W, tau_v, tau_I, v_th, t_first,
t_end, M, t_offset, and for conv stride, pad; penalty constants t_head_l,
t_tail_l, gamma_head, gamma_tail, gamma_q (missing = 0); optionally
skip = (src, delay): the skip-and-delay input of App. C.3 (Fig.
skip_connection), where the layer sees, along channels, the output of layer
src (-1 = the network input) delayed by `delay`, followed by the previous
layer's output.
Spike tensors: dense [B, N]; conv [B, C, H, W] (channel-major). A dense
layer after a conv layer flattens in (C, H, W) order.
"""

import numpy as np

from . import dstd, losses

INF = np.inf


def conv_out_hw(H, W, k, stride, pad):
    return (H + 2 * pad - k) // stride + 1, (W + 2 * pad - k) // stride + 1


def _pad_s(s, pad):
    if pad == 0:
        return s
    return np.pad(s, [(0, 0)] * (s.ndim - 2) + [(pad, pad), (pad, pad)])


def conv_what(s, Wc, stride, pad):
    """w^[b, o, y, x, m] = sum_{c,kh,kw} W[o,c,kh,kw] s[b, m, c, y s + kh - p, x s + kw - p].

    s [B, M, C, H, W] (zero outside the image: padding is silent input).
    """
    B, M, C, H, Wd = s.shape
    O, _, k, _ = Wc.shape
    Ho, Wo = conv_out_hw(H, Wd, k, stride, pad)
    sp = _pad_s(s, pad)
    out = np.zeros((B, O, Ho, Wo, M))
    for kh in range(k):
        for kw in range(k):
            patch = sp[:, :, :, kh:kh + stride * (Ho - 1) + 1:stride, kw:kw + stride * (Wo - 1) + 1:stride]
            out += np.einsum("bmcyx,oc->boyxm", patch, Wc[:, :, kh, kw])
    return out


def conv_what_adjoint(gw, s, Wc, stride, pad):
    """Adjoint of ``conv_what``: returns (g_W [O,C,k,k], g_s [B, M, C, H, W])."""
    B, M, C, H, Wd = s.shape
    O, _, k, _ = Wc.shape
    Ho, Wo = conv_out_hw(H, Wd, k, stride, pad)
    sp = _pad_s(s, pad)
    gsp = np.zeros_like(sp)
    gW = np.zeros_like(Wc, dtype=float)
    for kh in range(k):
        for kw in range(k):
            sl = (slice(None), slice(None), slice(None),
                  slice(kh, kh + stride * (Ho - 1) + 1, stride),
                  slice(kw, kw + stride * (Wo - 1) + 1, stride))
            patch = sp[sl]
            gW[:, :, kh, kw] = np.einsum("boyxm,bmcyx->oc", gw, patch)
            gsp[sl] += np.einsum("boyxm,oc->bmcyx", gw, Wc[:, :, kh, kw])
    if pad:
        gsp = gsp[..., pad:-pad, pad:-pad]
    return gW, gsp


def layer_grid(L):
    return dstd.grid(L["t_first"], L["t_end"], L["M"], L.get("t_offset", 0.0))


def forward_layer(t_in, L, solver="table"):
    """One layer of Alg. 2. Returns its context dict (t reshaped to the layer's output shape)."""
    T, dt = layer_grid(L)
    tv, ti, V = L["tau_v"], L["tau_I"], L["v_th"]
    W = np.asarray(L["W"], float)
    if L["kind"] == "dense":
        x = t_in.reshape(t_in.shape[0], -1)
        ctx = dstd.forward_dense(x, W, T, dt, tv, ti, V, solver)
        ctx["out_shape"] = ctx["t"].shape
    else:
        B, C, H, Wd = t_in.shape
        s = dstd.binning(t_in.reshape(B, -1), T, dt, tv, ti).reshape(B, L["M"], C, H, Wd)
        what = conv_what(s, W, L["stride"], L["pad"])
        Bo, O, Ho, Wo, M = what.shape
        ctx = dstd.solve(what.reshape(B, O * Ho * Wo, M), T, dt, tv, ti, V, solver)
        ctx.update(s=s, what=what)
        ctx["out_shape"] = (B, O, Ho, Wo)
    ctx["T"], ctx["dt"] = T, dt
    ctx["t_in"] = t_in
    for key in ("t", "q", "vpeak", "vdot", "fired"):
        ctx[key] = ctx[key].reshape(ctx["out_shape"])
    return ctx


def backward_layer(ctx, L, g_t):
    """Gradients of one layer: (g_W, g_t_in shaped like the layer input)."""
    T, dt = ctx["T"], ctx["dt"]
    tv, ti, V = L["tau_v"], L["tau_I"], L["v_th"]
    W = np.asarray(L["W"], float)
    t_in = ctx["t_in"]
    B = t_in.shape[0]
    flat = {k: ctx[k].reshape(B, -1) for k in ("t", "q", "vdot", "fired")}
    gw = dstd.solve_backward(flat, g_t.reshape(B, -1), T, dt, tv, ti, V)
    if L["kind"] == "dense":
        x = t_in.reshape(B, -1)
        g_W = np.einsum("bim,bmj->ij", gw, ctx["s"])
        gS = np.einsum("bim,ij->bmj", gw, W)
        ds = dstd.binning(x, T, dt, tv, ti, derivative=True)
        g_in = np.sum(gS * ds, axis=1).reshape(t_in.shape)
    else:
        _, O, Ho, Wo = ctx["out_shape"]
        gw5 = gw.reshape(B, O, Ho, Wo, -1)
        g_W, gs = conv_what_adjoint(gw5, ctx["s"], W, L["stride"], L["pad"])
        ds = dstd.binning(t_in.reshape(B, -1), T, dt, tv, ti, derivative=True).reshape(gs.shape)
        g_in = np.sum(gs * ds, axis=1)
    return g_W, g_in


def penalty_norm(ctx):
    """1/B for dense layers, 1/(B H_o W_o) for conv layers (App. C.1)."""
    shp = ctx["out_shape"]
    return 1.0 / (shp[0] * (shp[2] * shp[3] if len(shp) == 4 else 1))


def w_rowsum(L):
    W = np.asarray(L["W"], float)
    return W.reshape(W.shape[0], -1).sum(1)


def layer_input(t0, ctxs, l, L):
    """Input of layer l: the previous output, with a skip layer's delayed
    source placed first along channels (App. C.3: the third layer of a
    skip-and-delay block also receives the block's input, 2 tau_shift later)."""
    x = np.asarray(t0, float) if l == 0 else ctxs[l - 1]["t"]
    sk = L.get("skip")
    if sk is None:
        return x
    src, delay = sk
    a = np.asarray(t0, float) if src < 0 else ctxs[src]["t"]
    return np.concatenate([a + delay, x], axis=1)


def forward_net(t0, layers, solver="table"):
    ctxs = []
    for l, L in enumerate(layers):
        ctxs.append(forward_layer(layer_input(t0, ctxs, l, L), L, solver))
    return ctxs


def train_objective(t0, layers, labels, tau_soft, solver="table", backward=True):
    """Eq. cost_function on one mini-batch, and its gradients.

    Returns (C, parts, grads) with parts = dict(ce, T, Q) and grads a list of
    dC/dW^(l) (None when ``backward`` is False), plus the layer contexts.
    """
    ctxs = forward_net(t0, layers, solver)
    last = layers[-1]
    tL = ctxs[-1]["t"].reshape(ctxs[-1]["t"].shape[0], -1)
    ce, g = losses.ce_loss(tL, labels, tau_soft, t_silent=last["t_end"])
    Tsum, Qsum = 0.0, 0.0
    gT, counts = [], []
    for ctx, L in zip(ctxs, layers):
        nrm = penalty_norm(ctx)
        tv, gt = losses.temporal_penalty(ctx["t"], L.get("t_head_l", 0.0), L.get("t_tail_l", 0.0),
                                         L.get("gamma_head", 0.0), L.get("gamma_tail", 0.0), nrm)
        Tsum += tv
        gT.append(gt)
        t2 = ctx["t"].reshape(ctx["t"].shape[0], ctx["t"].shape[1], -1) if ctx["t"].ndim == 4 \
            else ctx["t"][..., None]
        # silent count per output channel (dense: per neuron)
        cnt = (~np.isfinite(t2)).sum((0, 2)).astype(float)
        counts.append(cnt)
        Qsum += -L.get("gamma_q", 0.0) * nrm * np.sum(cnt * w_rowsum(L))
    C = ce + Tsum + Qsum
    parts = {"ce": ce, "T": Tsum, "Q": Qsum}
    if not backward:
        return C, parts, None, ctxs
    grads = [None] * len(layers)
    # dC/d(output of layer l) from the layers that read it (and the loss)
    g_out = [np.zeros(c["t"].shape) for c in ctxs]
    g_out[-1] = g.reshape(ctxs[-1]["t"].shape)
    for l in range(len(layers) - 1, -1, -1):
        ctx, L = ctxs[l], layers[l]
        g_t = g_out[l] + gT[l]
        g_W, g_in = backward_layer(ctx, L, g_t)
        nrm = penalty_norm(ctx)
        W = np.asarray(L["W"], float)
        qg = -L.get("gamma_q", 0.0) * nrm * counts[l]
        g_W = g_W + qg.reshape((-1,) + (1,) * (W.ndim - 1))
        grads[l] = g_W
        sk = L.get("skip")
        if sk is not None:
            # split along channels; the delay has unit derivative
            src = sk[0]
            Ca = (np.asarray(t0).shape if src < 0 else ctxs[src]["t"].shape)[1]
            if src >= 0:
                g_out[src] = g_out[src] + g_in[:, :Ca]
            g_in = g_in[:, Ca:]
        if l > 0:
            g_out[l - 1] = g_out[l - 1] + g_in.reshape(ctxs[l - 1]["t"].shape)
    return C, parts, grads, ctxs


def e_rmse(t_exact, t_dstd):
    """E_RMSE of App. E.1 over the outputs where both methods fire, and the
    number of outputs whose firing state differs."""
    a = np.asarray(t_exact, float).ravel()
    b = np.asarray(t_dstd, float).ravel()
    both = np.isfinite(a) & np.isfinite(b)
    mism = int(np.sum(np.isfinite(a) != np.isfinite(b)))
    if not both.any():
        return np.nan, mism
    return float(np.sqrt(np.mean((a[both] - b[both]) ** 2))), mism
