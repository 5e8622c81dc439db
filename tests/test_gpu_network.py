"""GPU parity of whole networks (Alg. 2 layer loop + Eq. cost_function) and of
the runtime pieces: CUDA-graph replay, kernel timing, bounded waits.

The 784-800-800-10 workload is checked at its full batch of 256, in the
bench's launch configuration (x3 tensor-core split, M = 32), layer by layer
with teacher forcing: each oracle layer is fed the GPU's previous-layer
spike times, so a near-threshold flip upstream cannot propagate.
"""

import math

import numpy as np
import pytest
import torch

from helpers import f32, oracle_forward, rel_l2, well_conditioned
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


def _cfg2_net(math_mode="x3", batch=256, keep=None, offsets=None):
    from paper_2607_14672_gb300 import configs, net
    cfg = configs.config2(batch=batch)
    if offsets is not None:
        cfg = configs.with_offsets(cfg, offsets)
    t0 = cfg["inputs"](B=256)
    lab = cfg["labels"](B=256)
    if keep is not None:
        t0, lab = t0[keep], lab[keep]
    n = net.DenseNet(cfg, math_mode, batch=t0.shape[0])
    n.set_inputs(f32(t0), lab)
    return cfg, n, f32(t0), lab


def _teacher_forced_forward(n, t0):
    """Oracle layer l on the GPU's layer l-1 output; returns per-layer contexts."""
    ctxs = []
    x = t0
    for l, L in enumerate(n.layers):
        Lw = dict(L, W=f32(L["W"]))
        ctxs.append(oracle_forward(x, Lw["W"], Lw))
        x = host(n.t[l])
    return ctxs


@pytest.mark.parametrize("math_mode", ["x3", "f32"])
def test_cfg2_full_batch_teacher_forced(math_mode):
    from paper_2607_14672_gb300 import configs, dstd
    offsets = configs.draw_offsets(configs.config2()["layers"])
    cfg, n, t0, lab = _cfg2_net(math_mode, offsets=offsets)
    n.step()
    torch.cuda.synchronize()
    B = t0.shape[0]
    ctxs = _teacher_forced_forward(n, t0)
    ill = []
    for l, (ctx, L) in enumerate(zip(ctxs, n.layers)):
        tg = host(n.t[l])
        ok = well_conditioned(ctx, L["v_th"])
        ill.append(~ok)
        fo, fg = np.isfinite(ctx["t"]), np.isfinite(tg)
        assert not (ok & (fo != fg)).any(), f"layer {l + 1}: mask mismatch"
        both = ok & fo & fg
        err = np.abs(tg[both] - ctx["t"][both]).max()
        assert err <= 1e-4 * configs.t_max(L), f"layer {l + 1}: max |dt| {err:.2e}"
        assert both.sum() > 0.5 * tg.size
    # CE gradient of the output layer
    tL = host(n.t[-1])
    _, gL = olosses.ce_loss(tL, lab, cfg["tau_soft"], n.layers[-1]["t_end"])
    assert rel_l2(host(n.g[-1]), gL) <= 1e-5
    # backward, layer by layer with teacher forcing: both sides get the same
    # upstream gradient; neurons whose peak grazes the threshold get a total
    # gradient of zero on both sides (GPU: upstream = -dT/dt cancels the
    # layer's own penalty term; oracle: zero)
    g_up = host(n.g[-1])
    gW_buf = [torch.empty_like(w) for w in n.W]
    for l in range(len(n.layers) - 1, -1, -1):
        L, ctx = n.layers[l], ctxs[l]
        Wl = f32(L["W"])
        tg = host(n.t[l])
        _, pg = olosses.temporal_penalty(tg, L["t_head_l"], L["t_tail_l"], L["gamma_head"], L["gamma_tail"], 1.0 / B)
        _, gT = olosses.temporal_penalty(ctx["t"], L["t_head_l"], L["t_tail_l"], L["gamma_head"],
                                         L["gamma_tail"], 1.0 / B)
        g_gpu = np.where(ill[l], -pg, g_up)
        g_ora = np.where(ill[l], 0.0, g_up + gT)
        x_dev = n.layer_input(l)
        x = t0 if l == 0 else host(n.t[l - 1])
        g_in = torch.empty_like(x_dev) if l > 0 else None
        dstd.dense_bwd(x_dev, n.W[l], n.t[l], n.saved[l], torch.tensor(g_gpu, dtype=torch.float32, device="cuda"),
                       n.p[l], math_mode, g_in, gW_buf[l], n.workspace)
        torch.cuda.synchronize()
        gW, gin, _ = odstd.backward_dense(ctx, x, Wl, g_ora, ctx["T"], ctx["dt"], L["tau_v"], L["tau_I"], L["v_th"])
        _, cnt = olosses.dead_neuron_penalty(tg, Wl.sum(1), L["gamma_q"], 1.0 / B)
        gW = gW - L["gamma_q"] / B * cnt[:, None]
        assert rel_l2(host(gW_buf[l]), gW) <= 1e-3, f"layer {l + 1} dW"
        if l > 0:
            assert rel_l2(host(g_in), gin) <= 1e-3, f"layer {l + 1} dt_in"
            g_up = host(g_in)


def test_cfg2_objective_matches_free_running_oracle():
    from paper_2607_14672_gb300 import configs
    cfg, n, t0, lab = _cfg2_net("x3", keep=np.arange(64))
    n.step()
    torch.cuda.synchronize()
    layers = [dict(L, W=f32(L["W"])) for L in n.layers]
    C, parts, grads, ctxs = onet.train_objective(t0, layers, lab, cfg["tau_soft"], backward=False)
    assert abs(float(n.objective()) - C) <= 1e-3 * abs(C)
    pen = host(n.penalty)
    for l, ctx in enumerate(ctxs):
        assert abs(pen[l, 3] - np.isfinite(ctx["t"]).sum()) <= 0.002 * ctx["t"].size


def test_graph_replay_equals_eager():
    cfg, n, t0, lab = _cfg2_net("x3", batch=256)
    n.step()
    torch.cuda.synchronize()
    t_e = [host(x) for x in n.t]
    gW_e = [host(x) for x in n.gW]
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        n.step()
        torch.cuda.synchronize()
        with torch.cuda.graph(g, stream=s):
            n.step()
    for x in n.t + n.gW:
        x.zero_()
    g.replay()
    torch.cuda.synchronize()
    for a, b in zip(t_e, n.t):
        np.testing.assert_array_equal(a, host(b))
    # dW adds its split-K slices with fp32 atomics, in whatever order they
    # finish: equal to fp32 rounding, not bitwise
    for a, b in zip(gW_e, n.gW):
        assert np.abs(a - host(b)).max() <= 1e-5 * np.abs(a).max()


def test_kernel_timing_counts_launches():
    from paper_2607_14672_gb300 import dstd
    cfg, n, t0, lab = _cfg2_net("x3", batch=64, keep=np.arange(64))
    n.step()
    dstd.timing_enable(True)
    for _ in range(3):
        n.step()
    tm = dstd.timing_read()
    dstd.timing_enable(False)
    # the 800 -> 10 readout runs on CUDA cores, one kernel each way (few outputs)
    assert tm["gemm_fwd_scan"][1] == 6 and tm["gemm_dW"][1] == 6 and tm["gemm_dS_gradt"][1] == 3
    assert tm["narrow_fwd"][1] == 3 and tm["narrow_bwd"][1] == 3 and tm["gradt_gather"][1] == 0
    assert sum(c for _, c in tm.values()) == 3 * n.launches_per_step()
    assert all(ms > 0 for ms, c in tm.values() if c > 0)


def test_kernel_timing_inside_a_graph():
    """Timing on while a step is captured: every launch gets event-record
    nodes in the graph, and each replay's kernel times are collected."""
    from paper_2607_14672_gb300 import dstd
    cfg, n, t0, lab = _cfg2_net("x3", batch=64, keep=np.arange(64))
    n.step()
    torch.cuda.synchronize()
    dstd.timing_enable(True)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            n.step()
        for _ in range(3):
            g.replay()
            dstd.timing_collect()
    tm = dstd.timing_read()
    dstd.timing_enable(False)
    assert sum(c for _, c in tm.values()) == 3 * n.launches_per_step()
    assert all(ms > 0 for ms, c in tm.values() if c > 0)
    assert tm["gemm_fwd_scan"][1] == 6 and tm["narrow_bwd"][1] == 3


def test_bounded_wait_reports_timeout():
    from paper_2607_14672_gb300 import dstd
    assert dstd.device_status(clear=True) == 0
    dstd.selftest_wait_timeout(20000)          # 20 ms wait on a barrier nothing completes
    assert dstd.device_status(clear=True) == -5
    # the context is still usable afterwards
    cfg, n, t0, lab = _cfg2_net("x3", batch=16, keep=np.arange(16))
    n.step()
    assert dstd.device_status(clear=True) == 0
    assert np.isfinite(float(n.objective()))


@pytest.mark.parametrize("N,M", [(1024, 32), (1024, 8), (4096, 128)])
def test_cfg3_single_layer(N, M):
    from paper_2607_14672_gb300 import configs, net
    cfg = configs.config3(N, M, batch=16)
    n = net.DenseNet(cfg, "x3", batch=16)
    t0 = f32(cfg["inputs"](B=16))
    n.set_inputs(t0)
    n.forward()
    torch.cuda.synchronize()
    L = dict(cfg["layers"][0], W=f32(cfg["layers"][0]["W"]))
    sel = np.arange(0, N, max(1, N // 512))          # sampled output neurons
    ctx = oracle_forward(t0, L["W"][sel], L)
    tg = host(n.t[0])[:, sel]
    ok = well_conditioned(ctx, 1.0)
    assert not (ok & (np.isfinite(ctx["t"]) != np.isfinite(tg))).any()
    both = ok & np.isfinite(ctx["t"]) & np.isfinite(tg)
    assert both.sum() > 0.3 * tg.size
    assert np.abs(tg[both] - ctx["t"][both]).max() <= 1e-4 * configs.t_max(L)


def test_cfg3_full_size_sampled():
    # N = 16384, B = 128, M = 128: the largest single-layer workload, checked on
    # sampled outputs the oracle computes one by one
    from paper_2607_14672_gb300 import configs, net
    cfg = configs.config3(16384, 128)
    n = net.DenseNet(cfg, "x3")
    t0 = f32(cfg["inputs"]())
    n.set_inputs(t0)
    n.forward()
    torch.cuda.synchronize()
    L = dict(cfg["layers"][0])
    g = np.random.default_rng(0)
    rows = g.choice(16384, 64, replace=False)
    bs = g.choice(128, 4, replace=False)
    ctx = oracle_forward(t0[bs], f32(L["W"][rows]), L)
    tg = host(n.t[0])[np.ix_(bs, rows)]
    ok = well_conditioned(ctx, 1.0)
    assert not (ok & (np.isfinite(ctx["t"]) != np.isfinite(tg))).any()
    both = ok & np.isfinite(ctx["t"]) & np.isfinite(tg)
    assert both.sum() > 64
    assert np.abs(tg[both] - ctx["t"][both]).max() <= 1e-4 * configs.t_max(L)


@pytest.mark.parametrize("math_mode", ["x3", "bf16"])
def test_cfg3_backward_full_size_sampled(math_mode):
    """N = 16384, B = 128, M = 128, sum-of-times loss: the backward in the
    launch configuration the bench times (dW on SM pairs, the cost model's
    pick at this width; dS with the input-time gradient in the contraction's
    epilogue; several persistent rounds of tiles). Checked against oracle
    steps on 8 sampled rows of dW (each a sum over every sample) and on the
    whole input-time gradient of 2 samples, within 1e-3 relative L2. bf16 runs
    the oracle on bf16-rounded contraction operands (reading R9). The oracle's
    backward runs at the GPU's spike state (the forward tests hold it to the
    tolerance)."""
    from paper_2607_14672_gb300 import configs, dstd, net
    from helpers import bf16, bf16_ambiguous_ulp, bf16_grad_rel_bound, decode_saved
    N, M = 16384, 128
    cfg = configs.config3(N, M)
    n = net.DenseNet(cfg, math_mode)
    t0 = f32(cfg["inputs"]())
    n.set_inputs(t0)
    B = n.B
    g_in = torch.empty(B, N, dtype=torch.float32, device="cuda")
    dstd.dense_fwd(n.t_in, n.W[0], n.p[0], math_mode, n.t[0], n.saved[0], n.penalty[0], n.workspace, None)
    dstd.sum_t_loss(n.t[0], n.loss, n.g[0], None)
    dstd.dense_bwd(n.t_in, n.W[0], n.t[0], n.saved[0], n.g[0], n.p[0], math_mode, g_in, n.gW[0], n.workspace, None)
    torch.cuda.synchronize()
    assert dstd.device_status(clear=True) == 0
    L = dict(cfg["layers"][0])
    W = f32(L["W"])
    rnd = bf16 if math_mode == "bf16" else (lambda a: a)
    Wr = rnd(W)
    T, dt = odstd.grid(L["t_first"], L["t_end"], M, L["t_offset"])
    tv, ti = L["tau_v"], L["tau_I"]
    tg = host(n.t[0])
    qg, _, vdg = decode_saved(n.saved[0].cpu().numpy(), B, N)

    def state(b, cols):
        """The GPU's spike state of sample b's neurons cols (held to the
        tolerance by the forward tests): the input-time gradient magnifies
        spike-time differences by about T / dt, so the backward is compared
        at the same state."""
        t = tg[b][cols][None]
        return {"t": t, "q": qg[b][cols][None].astype(int), "vdot": vdg[b][cols][None], "fired": np.isfinite(t)}

    # dW rows: every sample's contribution
    g = np.random.default_rng(3)
    rows = np.sort(g.choice(N, 8, replace=False))
    # bf16: dw^ entries at a rounding midpoint may round either way (helpers.bf16_grad_rel_bound)
    amb = (lambda a: bf16_ambiguous_ulp(a, 2.0 ** -16)) if math_mode == "bf16" else (lambda a: np.zeros_like(a))
    gW_ref = np.zeros((len(rows), N))
    bW = np.zeros((len(rows), N))
    for b in range(B):
        sr = rnd(odstd.binning(t0[b], T, dt, tv, ti))                     # [M, N]
        ctx = state(b, rows)
        gw = odstd.solve_backward(ctx, ctx["fired"].astype(float), T, dt, tv, ti, 1.0)[0]   # [8, M]
        gW_ref += rnd(gw) @ sr
        bW += amb(gw) @ np.abs(sr)
    e_w = rel_l2(host(n.gW[0])[rows], gW_ref)
    assert e_w <= 1e-3 + bf16_grad_rel_bound(bW, gW_ref), e_w
    # input-time gradient of two whole samples: every neuron's dw^, then W^T
    for b in (0, B - 1):
        ctx = state(b, slice(None))
        gw = odstd.solve_backward(ctx, ctx["fired"].astype(float), T, dt, tv, ti, 1.0)[0]    # [N, M]
        dS = rnd(gw).T @ Wr                                                # [M, N]
        ds = odstd.binning(t0[b], T, dt, tv, ti, derivative=True)
        ref = np.sum(dS * ds, axis=0)
        bnd = np.sum((amb(gw).T @ np.abs(Wr)) * np.abs(ds), axis=0) if math_mode == "bf16" else 0.0 * ref
        e_g, a_g = rel_l2(host(g_in)[b], ref), bf16_grad_rel_bound(bnd, ref)
        assert e_g <= 1e-3 + a_g, (b, e_g, a_g)
