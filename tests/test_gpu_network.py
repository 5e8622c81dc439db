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
