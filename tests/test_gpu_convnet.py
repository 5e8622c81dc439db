"""GPU parity of the convolutional networks (configs 4 and 5) against the
float64 oracle, in bf16 (the workloads' precision).

The GPU runs whole training steps (forward, CE + T + Q, backward, AdamW).
Parity is checked layer by layer with teacher forcing (each oracle layer is
fed the GPU's input to that layer), on the oracle run with bf16-rounded
contraction operands (reading R9):

* config 4 (tau = (inf, inf), closed-form solve), full batch: every neuron of
  two images of every layer, plus a free-running oracle pass of those images
  whose per-layer firing fractions must agree;
* config 5 (tau = (1.0, 0.25), numeric solve), full batch: 192 sampled
  neurons per layer, each recomputed from its 3x3 receptive field, and the
  per-layer silent (dead) share on those neurons;
* gradients of both networks at full width (batch 4): for every conv layer,
  the weight gradient of one output channel (a sum over every position of
  every image) and the input-time gradient of every channel at two input
  positions, each within 1e-3 relative L2 of the oracle's backward at the
  GPU's spike state (held to the tolerance by the forward checks), plus the
  allowance for dC/dw^ entries at a bf16 rounding midpoint
  (``helpers.bf16_grad_rel_bound``).

Spike times meet |dt| <= 1e-4 T_max and masks agree outside the 1e-5 band
around the threshold, except where a neuron's own bound on the bf16
difference allows more (``helpers.check_bf16_times``): a grid weight that
lies within a few fp32 ulps of a bf16 rounding midpoint may round to the
other neighbour on the GPU (fp32) than in the oracle (float64), and the
tensor core accumulates the exact bf16 products in fp32.
"""

import math

import numpy as np
import pytest
import torch

from helpers import (bf16, bf16_ambiguous_ulp, bf16_grad_rel_bound, check_bf16_times, conv_neurons, decode_saved,
                     dense_bound_fn, grid_of, neuron_bound_fn, oracle_forward, rel_l2)
from oracle import dstd as odstd, losses as olosses, network as onet

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2607_14672_gb300 import build, dstd
    build.build()
    dstd.load()
    assert dstd.device_status(clear=True) == 0
    yield
    assert dstd.device_status(clear=True) == 0


def host(x):
    return x.detach().cpu().numpy().astype(np.float64)


def to_nchw(t):
    return t.transpose(0, 3, 1, 2) if t.ndim == 4 else t


def run_net(cfg):
    from paper_2607_14672_gb300 import configs, net
    cfg = configs.with_offsets(cfg, configs.draw_offsets(cfg["layers"]))
    n = net.ConvNet(cfg)
    t0 = cfg["inputs"]()
    lab = cfg["labels"]()
    n.set_inputs(t0.astype(np.float32), lab)
    n.step()
    torch.cuda.synchronize()
    from paper_2607_14672_gb300 import dstd
    assert dstd.device_status(clear=True) == 0
    return cfg, n, np.asarray(t0, np.float32).astype(np.float64), lab


def oracle_conv_layer(x, L, operand_round=bf16):
    """Oracle conv layer on bf16-rounded s and W; x [B, C, H, W]."""
    T, dt = grid_of(L)
    tv, ti, V = L["tau_v"], L["tau_I"], L["v_th"]
    B, C, H, Wd = x.shape
    s = odstd.binning(x.reshape(B, -1), T, dt, tv, ti).reshape(B, L["M"], C, H, Wd)
    what = onet.conv_what(operand_round(s), operand_round(np.asarray(L["W"], np.float32)), L["stride"], L["pad"])
    _, O, Ho, Wo, M = what.shape
    ctx = odstd.solve(what.reshape(B, O * Ho * Wo, M), T, dt, tv, ti, V)
    out = {k: ctx[k].reshape(B, O, Ho, Wo) for k in ("t", "vpeak", "q", "vdot", "fired")}
    out["T"], out["dt"] = T, dt
    return out


def conv_layer_bound_fn(x, ctx, L):
    """Per-neuron bf16 bound of a whole-layer oracle context (receptive fields of the flagged neurons only)."""
    from helpers import bf16_potential_bound, kernel_max
    shape = ctx["t"].shape
    kmax = kernel_max(ctx["T"], L["tau_v"], L["tau_I"])

    def fn(idx):
        b, o, y, xx = np.unravel_index(idx, shape)
        nc = conv_neurons(x, L, list(zip(b, o, y, xx)))
        return bf16_potential_bound(nc["s"], nc["w"], ctx["q"].ravel()[idx], ctx["t"].ravel()[idx], ctx["T"],
                                    L["tau_v"], L["tau_I"], kmax)
    return fn


def compare_layer(t_gpu, ctx, L, bound_fn, min_cmp=0.9):
    n_cmp, n_bound = check_bf16_times(t_gpu, ctx, L, bound_fn)
    ok = np.abs(np.asarray(ctx["vpeak"]) - L["v_th"]) > 1e-5
    assert ok.sum() > min_cmp * np.asarray(t_gpu).size
    assert n_bound <= 0.01 * np.asarray(t_gpu).size
    return n_cmp


def dense_readout_ctx(x, L):
    W = np.asarray(L["W"], np.float32).astype(np.float64)
    ctx = oracle_forward(x.reshape(x.shape[0], -1), W, L, operand_round=bf16)
    return ctx, dense_bound_fn(ctx, W, L)


def test_cfg4_conv_network_layers_match_oracle():
    from paper_2607_14672_gb300 import configs
    cfg, n, t0, lab = run_net(configs.config4())
    imgs = [0, n.B - 1]
    x = t0[imgs]
    for l, L in enumerate(cfg["layers"]):
        t_gpu = to_nchw(host(n.t[l]))[imgs]
        if L["kind"] == "conv":
            ctx = oracle_conv_layer(x, L)
            fn = conv_layer_bound_fn(x, ctx, L)
        else:
            ctx, fn = dense_readout_ctx(x, L)
        compare_layer(t_gpu, ctx, L, fn)
        x = t_gpu                                   # teacher forcing: next layer sees the GPU's output
    # every layer fires, and the whole batch's dead share is recorded by the counters
    dead = n.dead_fraction()
    assert all(0.0 <= d < 1.0 for d in dead)
    for g in n.gW:
        assert torch.isfinite(g).all()


def test_cfg4_free_running_firing_matches_oracle():
    # free-running oracle (no GPU input) on two images: per-layer firing shares
    from paper_2607_14672_gb300 import configs
    cfg, n, t0, lab = run_net(configs.config4())
    imgs = [0, 1]
    x = t0[imgs]
    for l, L in enumerate(cfg["layers"][:-1]):
        ctx = oracle_conv_layer(x, L)
        f_ora = np.isfinite(ctx["t"]).mean()
        f_gpu = np.isfinite(to_nchw(host(n.t[l]))[imgs]).mean()
        assert abs(f_ora - f_gpu) <= 0.01, (l, f_ora, f_gpu)
        x = ctx["t"]


def test_cfg5_conv_network_sampled_neurons_match_oracle():
    from paper_2607_14672_gb300 import configs
    cfg, n, t0, lab = run_net(configs.config5())
    rng = np.random.default_rng(5)
    imgs = [0, n.B - 1]
    x_all = t0
    for l, L in enumerate(cfg["layers"]):
        t_gpu = to_nchw(host(n.t[l]))
        x = x_all[imgs]
        if L["kind"] == "conv":
            _, O, Ho, Wo = t_gpu.shape
            idx = [(bi, int(rng.integers(O)), int(rng.integers(Ho)), int(rng.integers(Wo)))
                   for bi in range(len(imgs)) for _ in range(96)]
            ctx = conv_neurons(x, L, idx)
            fn = neuron_bound_fn(ctx, L)
            tg = np.array([t_gpu[imgs[b], o, y, xx] for (b, o, y, xx) in idx])
        else:
            ctx, fn = dense_readout_ctx(x, L)
            tg = t_gpu[imgs]
        compare_layer(tg, ctx, L, fn)
        # dead (silent) share on the sampled neurons, away from the threshold
        okm = np.abs(ctx["vpeak"] - L["v_th"]) > 1e-5
        assert abs(np.mean(~np.isfinite(tg[okm])) - np.mean(~np.isfinite(ctx["t"][okm]))) <= 2.0 / okm.sum()
        x_all = t_gpu                               # teacher forcing
    for g in n.gW:
        assert torch.isfinite(g).all()


# ---------------------------------------------------------------------------
# gradients at full width (every conv layer of configs 4 and 5, batch 4)
# ---------------------------------------------------------------------------
def gpu_state(n, l):
    """The GPU's spike state of layer l as [B, O, Ho, Wo] arrays (t, q, dv^/dt)."""
    t = host(n.t[l])
    B, Ho, Wo, O = t.shape
    q, _, vd = decode_saved(n.saved[l].cpu().numpy(), B * Ho * Wo, O)
    tr = lambda a: np.asarray(a, float).reshape(B, Ho, Wo, O).transpose(0, 3, 1, 2)
    return to_nchw(t), tr(q), tr(vd)


def oracle_dW_row(x, L, o, g_up, gstate, nrm):
    """dC/dW[o] of a conv layer (oracle steps on bf16-rounded operands) at the
    GPU's spike state of output channel o (every position of every image):
    the IFT backward with the upstream gradient plus T', the adjoint
    contraction, and the dead-neuron term. The state itself is held to the
    tolerance by the forward checks; the input-time gradient would magnify
    its legitimate bf16 differences (a difference of dS at adjacent grid
    points), so both gradients are compared at the same state."""
    T, dt = grid_of(L)
    tv, ti, V = L["tau_v"], L["tau_I"], L["v_th"]
    B, C, H, Wd = x.shape
    W = np.asarray(L["W"], np.float32).astype(np.float64)[o:o + 1]
    s = odstd.binning(x.reshape(B, -1), T, dt, tv, ti).reshape(B, L["M"], C, H, Wd)
    tg, qg, vdg = (a[:, o] for a in gstate)
    _, _, Ho, Wo = gstate[0].shape
    _, gT = olosses.temporal_penalty(tg, L["t_head_l"], L["t_tail_l"], L["gamma_head"], L["gamma_tail"], nrm)
    flat = {"t": tg.reshape(B, -1), "q": qg.reshape(B, -1).astype(int), "vdot": vdg.reshape(B, -1),
            "fired": np.isfinite(tg).reshape(B, -1)}
    gw = odstd.solve_backward(flat, (g_up[:, o] + gT).reshape(B, -1), T, dt, tv, ti, V)
    gw5 = gw.reshape(B, 1, Ho, Wo, -1)
    gW, _ = onet.conv_what_adjoint(bf16(gw5), bf16(s), bf16(W), L["stride"], L["pad"])
    bW, _ = onet.conv_what_adjoint(bf16_ambiguous_ulp(gw5, 2.0 ** -16), np.abs(bf16(s)), np.abs(bf16(W)),
                                   L["stride"], L["pad"])
    cnt = float((~np.isfinite(tg)).sum())
    return gW[0] - L["gamma_q"] * nrm * cnt, bW[0]


def oracle_input_grad(x, L, b, yi, xi, g_up, gstate, nrm):
    """dC/dt_in of every channel of input position (b, yi, xi), at the GPU's
    spike state of the output neurons whose receptive field holds it (all
    channels): their IFT backward, then sum_m (sum_o W dw^) ds/dt (the
    derivative of Tab. DSTD_kernels), on bf16-rounded W and dw^."""
    T, dt = grid_of(L)
    tv, ti, V = L["tau_v"], L["tau_I"], L["v_th"]
    W = np.asarray(L["W"], np.float32).astype(np.float64)
    O, C, k, _ = W.shape
    st, pad = L["stride"], L["pad"]
    _, _, Ho, Wo = gstate[0].shape
    taps = [(y, xx, yi - y * st + pad, xi - xx * st + pad) for y in range(Ho) for xx in range(Wo)
            if 0 <= yi - y * st + pad < k and 0 <= xi - xx * st + pad < k]
    g = np.stack([g_up[b, :, y, xx] for (y, xx, _, _) in taps])           # [P, O]
    tg, qg, vdg = (np.stack([a[b, :, y, xx] for (y, xx, _, _) in taps]) for a in gstate)
    _, gT = olosses.temporal_penalty(tg, L["t_head_l"], L["t_tail_l"], L["gamma_head"], L["gamma_tail"], nrm)
    ctx = {"t": tg, "q": qg.astype(int), "vdot": vdg, "fired": np.isfinite(tg)}
    gw64 = odstd.solve_backward(ctx, g + gT, T, dt, tv, ti, V)              # [P, O, M]
    gw, amb = bf16(gw64), bf16_ambiguous_ulp(gw64, 2.0 ** -16)
    dS = sum(bf16(W[:, :, kh, kw]).T @ gw[p] for p, (_, _, kh, kw) in enumerate(taps))   # [C, M]
    bS = sum(np.abs(bf16(W[:, :, kh, kw])).T @ amb[p] for p, (_, _, kh, kw) in enumerate(taps))
    ds = odstd.binning(x[b, :, yi, xi], T, dt, tv, ti, derivative=True)    # [M, C]
    return np.sum(dS * ds.T, axis=1), np.sum(bS * np.abs(ds.T), axis=1)


def check_network_gradients(cfg, seed):
    from paper_2607_14672_gb300 import dstd
    cfg, n, t0, lab = run_net(cfg)
    rng = np.random.default_rng(seed)
    B = n.B
    worst = []
    for l, L in enumerate(cfg["layers"]):
        if L["kind"] != "conv":
            continue
        x = to_nchw(host(n.layer_input(l)))
        g_up = to_nchw(host(n.g[l]))
        gstate = gpu_state(n, l)
        _, O, Ho, Wo = gstate[0].shape
        nrm = 1.0 / (B * Ho * Wo)
        o = int(rng.integers(O))
        ref, bnd = oracle_dW_row(x, L, o, g_up, gstate, nrm)
        got = host(n.gW[l])[o].transpose(2, 0, 1)                          # [k, k, C] -> [C, k, k]
        e_w, a_w = rel_l2(got, ref), bf16_grad_rel_bound(bnd, ref)
        assert e_w <= 1e-3 + a_w, (l, o, e_w, a_w)
        if l == 0:
            worst.append((l, e_w, a_w))
            continue
        H, Wd = x.shape[2], x.shape[3]
        got_g, ref_g, bnd_g = [], [], []
        for (b, yi, xi) in [(0, 0, 0), (B - 1, int(rng.integers(1, H - 1)), int(rng.integers(1, Wd - 1)))]:
            ref, bnd = oracle_input_grad(x, L, b, yi, xi, g_up, gstate, nrm)
            ref_g.append(ref)
            bnd_g.append(bnd)
            got_g.append(to_nchw(host(n.g[l - 1]))[b, :, yi, xi])
        ref_g = np.concatenate(ref_g)
        e_g, a_g = rel_l2(np.concatenate(got_g), ref_g), bf16_grad_rel_bound(np.concatenate(bnd_g), ref_g)
        assert e_g <= 1e-3 + a_g, (l, e_g, a_g)
        worst.append((l, e_w, a_w, e_g, a_g))
    assert dstd.device_status(clear=True) == 0
    return worst


def test_cfg4_gradients_full_width_match_oracle():
    from paper_2607_14672_gb300 import configs
    print(check_network_gradients(configs.config4(batch=4), 41))


def test_cfg5_gradients_full_width_match_oracle():
    from paper_2607_14672_gb300 import configs
    print(check_network_gradients(configs.config5(batch=4), 51))


@pytest.mark.parametrize("shape,tau,seed", [((64, 16, 128, 1), (math.inf, math.inf), 4),
                                            ((128, 14, 128, 1), (1.0, 0.25), 5),
                                            ((64, 28, 128, 2), (1.0, 0.25), 6)])
def test_conv_backward_at_network_constants(shape, tau, seed):
    """Conv backward (x3) against the oracle on layer shapes and tau of configs 4 and 5."""
    from paper_2607_14672_gb300 import dstd
    from helpers import rel_l2
    C, H, O, stride = shape
    g = np.random.default_rng(seed)
    B = 1
    t = np.where(g.random((B, C, H, H)) < 0.1, np.inf, g.uniform(0.0, 1.0, (B, C, H, H))).astype(np.float32)
    wmean = {(math.inf, math.inf): 0.0052, (1.0, 0.25): 0.03}[tau] * 64 / C
    W = g.normal(wmean, 1.0 / math.sqrt(C * 9), (O, C, 3, 3)).astype(np.float32)
    L = dict(kind="conv", W=W.astype(np.float64), tau_v=tau[0], tau_I=tau[1], v_th=1.0, t_first=0.0, t_end=1.2,
             M=32 if tau[0] == math.inf else 64, t_offset=0.004, stride=stride, pad=1, t_head_l=0.35,
             t_tail_l=0.8, gamma_head=0.05, gamma_tail=0.01, gamma_q=1e-3)
    Ho, Wo = dstd.conv_out_hw(H, H, 3, stride, 1)
    p = dstd.params(L, 1.0 / (B * Ho * Wo))
    ws = torch.empty(dstd.conv_workspace_bytes(B, H, H, C, O, 3, stride, 1, p, "x3"), dtype=torch.uint8,
                     device="cuda")
    t_in = torch.tensor(t.transpose(0, 2, 3, 1).copy(), device="cuda")
    Wg = torch.tensor(W.transpose(0, 2, 3, 1).copy(), device="cuda")
    t_out = torch.empty(B, Ho, Wo, O, device="cuda")
    saved = torch.empty(dstd.dense_saved_bytes(B * Ho * Wo, O), dtype=torch.uint8, device="cuda")
    pen = torch.empty(4, device="cuda")
    dstd.conv_fwd(t_in, Wg, stride, 1, p, "x3", t_out, saved, pen, ws)
    torch.cuda.synchronize()
    ctx = onet.forward_layer(t.astype(np.float64), L)
    tg = host(t_out).transpose(0, 3, 1, 2)
    ok = np.abs(ctx["vpeak"] - 1.0) > 1e-5
    assert not (ok & (np.isfinite(tg) != np.isfinite(ctx["t"]))).any()
    assert np.isfinite(tg).mean() > 0.2
    up = g.normal(0.0, 1.0, ctx["t"].shape)
    from oracle import losses as olosses
    _, pg = olosses.temporal_penalty(tg, 0.35, 0.8, 0.05, 0.01, 1.0 / (B * Ho * Wo))
    _, gT = olosses.temporal_penalty(ctx["t"], 0.35, 0.8, 0.05, 0.01, 1.0 / (B * Ho * Wo))
    g_gpu = np.where(~ok, -pg, up)
    g_ora = np.where(~ok, 0.0, up + gT)
    g_t_in = torch.empty_like(t_in)
    g_W = torch.empty_like(Wg)
    dstd.conv_bwd(t_in, Wg, t_out, saved, torch.tensor(g_gpu.transpose(0, 2, 3, 1).copy(), dtype=torch.float32,
                                                       device="cuda"),
                  stride, 1, p, "x3", g_t_in, g_W, ws)
    torch.cuda.synchronize()
    gW, gin = onet.backward_layer(ctx, L, g_ora)
    cnt = (~np.isfinite(tg)).sum((0, 2, 3))
    gW = gW - 1e-3 / (B * Ho * Wo) * cnt[:, None, None, None]
    assert rel_l2(host(g_W).transpose(0, 3, 1, 2), gW) <= 1e-3
    assert rel_l2(host(g_t_in).transpose(0, 3, 1, 2), gin) <= 1e-3
