"""GPU parity of the convolutional DSTD layer against the float64 oracle.

The oracle's conv layer works channel-major (t [B, C, H, W], W [O, C, k, k]);
the library works NHWC (t [B, H, W, C], W [O, k, k, C]); the tests transpose.
Tolerances as for dense layers: |dt| <= 1e-4 T_max with masks identical
outside the 1e-5 near-threshold band, gradients to 1e-3 relative L2.
"""

import math

import numpy as np
import pytest
import torch

from helpers import f32, rel_l2
from oracle import dstd as odstd, losses as olosses, network as onet

pytestmark = pytest.mark.gpu

INF = math.inf


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2607_14672_gb300 import build, dstd
    build.build()
    dstd.load()
    assert dstd.device_status(clear=True) == 0
    yield
    assert dstd.device_status(clear=True) == 0


def dev(x):
    return torch.tensor(np.ascontiguousarray(x), dtype=torch.float32, device="cuda")


def host(x):
    return x.detach().cpu().numpy().astype(np.float64)


def conv_case(B, C, H, O, k, stride, pad, M, tau, seed, wmean, gammas=(0.0, 0.0, 0.0), silent=0.3, t_offset=0.011):
    g = np.random.default_rng(seed)
    t = f32(np.where(g.random((B, C, H, H)) < silent, INF, g.uniform(0, 1, (B, C, H, H))))
    W = f32(g.normal(wmean, 1.0 / math.sqrt(C * k * k), (O, C, k, k)))
    L = dict(kind="conv", W=W, tau_v=tau[0], tau_I=tau[1], v_th=1.0, t_first=0.0, t_end=1.2, M=M, t_offset=t_offset,
             stride=stride, pad=pad, t_head_l=0.35, t_tail_l=0.8, gamma_head=gammas[0], gamma_tail=gammas[1],
             gamma_q=gammas[2])
    return t, L


def run_conv_fwd(t, L, math_mode="x3"):
    from paper_2607_14672_gb300 import dstd
    B, C, H, Wd = t.shape
    O, _, k, _ = L["W"].shape
    Ho, Wo = dstd.conv_out_hw(H, Wd, k, L["stride"], L["pad"])
    p = dstd.params(L, 1.0 / (B * Ho * Wo))
    ws = torch.empty(dstd.conv_workspace_bytes(B, H, Wd, C, O, k, L["stride"], L["pad"], p, math_mode),
                     dtype=torch.uint8, device="cuda")
    t_in = dev(t.transpose(0, 2, 3, 1))
    Wg = dev(L["W"].transpose(0, 2, 3, 1))
    t_out = torch.empty(B, Ho, Wo, O, device="cuda")
    saved = torch.empty(dstd.dense_saved_bytes(B * Ho * Wo, O), dtype=torch.uint8, device="cuda")
    pen = torch.empty(4, device="cuda")
    dstd.conv_fwd(t_in, Wg, L["stride"], L["pad"], p, math_mode, t_out, saved, pen, ws)
    torch.cuda.synchronize()
    return dict(t=host(t_out).transpose(0, 3, 1, 2), t_in=t_in, W=Wg, t_out=t_out, saved=saved, pen=host(pen), p=p,
                ws=ws)


def check(t_gpu, ctx, L):
    ok = np.abs(ctx["vpeak"] - L["v_th"]) > 1e-5
    fo, fg = np.isfinite(ctx["t"]), np.isfinite(t_gpu)
    assert not (ok & (fo != fg)).any()
    both = ok & fo & fg
    assert both.sum() > 0.2 * t_gpu.size
    assert np.abs(t_gpu[both] - ctx["t"][both]).max() <= 1e-4 * (L["t_end"] - L["t_first"])
    return ok


# weight means giving about 60% firing with 64 input channels (scaled by 64/C)
WMEAN64 = {(0.5, 0.25): 0.035, (INF, INF): 0.0052, (1.0, 0.25): 0.024}


@pytest.mark.parametrize("tau", [(0.5, 0.25), (INF, INF), (1.0, 0.25)])
@pytest.mark.parametrize("C,H,O,stride", [(64, 8, 48, 1), (64, 9, 64, 2), (3, 12, 64, 1), (128, 6, 130, 1)])
def test_conv_forward_matches_oracle(tau, C, H, O, stride):
    t, L = conv_case(2, C, H, O, 3, stride, 1, 32, tau, seed=C + H, wmean=WMEAN64[tau] * 64 / C)
    r = run_conv_fwd(t, L)
    ctx = onet.forward_layer(t, L)
    check(r["t"], ctx, L)


def test_conv_backward_matches_oracle():
    from paper_2607_14672_gb300 import dstd
    t, L = conv_case(2, 64, 8, 48, 3, 1, 1, 32, (0.5, 0.25), seed=3, wmean=0.035, gammas=(0.05, 0.01, 1e-3))
    r = run_conv_fwd(t, L)
    ctx = onet.forward_layer(t, L)
    ok = check(r["t"], ctx, L)
    B, O, Ho, Wo = ctx["t"].shape
    nrm = 1.0 / (B * Ho * Wo)
    g = np.random.default_rng(4).normal(0.0, 1.0, ctx["t"].shape)
    ill = ~ok
    tg = r["t"]
    _, pg = olosses.temporal_penalty(tg, 0.35, 0.8, 0.05, 0.01, nrm)
    _, gT = olosses.temporal_penalty(ctx["t"], 0.35, 0.8, 0.05, 0.01, nrm)
    g_gpu = np.where(ill, -pg, g)
    g_ora = np.where(ill, 0.0, g + gT)
    g_t_in = torch.empty_like(r["t_in"])
    g_W = torch.empty_like(r["W"])
    dstd.conv_bwd(r["t_in"], r["W"], r["t_out"], r["saved"], dev(g_gpu.transpose(0, 2, 3, 1)), 1, 1, r["p"], "x3",
                  g_t_in, g_W, r["ws"])
    torch.cuda.synchronize()
    gW, gin = onet.backward_layer(ctx, L, g_ora)
    cnt = (~np.isfinite(tg)).sum((0, 2, 3))
    gW = gW - 1e-3 * nrm * cnt[:, None, None, None]
    assert rel_l2(host(g_W).transpose(0, 3, 1, 2), gW) <= 1e-3
    assert rel_l2(host(g_t_in).transpose(0, 3, 1, 2), gin) <= 1e-3


def test_conv_chunked_matches_unchunked():
    # 32 images of 32x32x64 at M = 32 exceed one ~1 GiB im2col chunk; the
    # result must not depend on where the chunks fall.
    from paper_2607_14672_gb300 import dstd
    t, L = conv_case(32, 64, 32, 64, 3, 1, 1, 32, (INF, INF), seed=9, wmean=0.0052)
    full = run_conv_fwd(t, L)
    parts = [run_conv_fwd(t[i:i + 8], L) for i in range(0, 32, 8)]
    tp = np.concatenate([q["t"] for q in parts], 0)
    np.testing.assert_array_equal(np.isfinite(full["t"]), np.isfinite(tp))
    fin = np.isfinite(tp)
    assert np.abs(full["t"][fin] - tp[fin]).max() <= 1e-6
    # weight gradient is a sum over images (no penalty terms here)
    g = np.where(np.isfinite(full["t"]), 1.0, 0.0)
    gWs = []
    for r, sl in [(full, slice(0, 32))] + [(q, slice(i, i + 8)) for q, i in zip(parts, range(0, 32, 8))]:
        g_W = torch.empty_like(r["W"])
        dstd.conv_bwd(r["t_in"], r["W"], r["t_out"], r["saved"], dev(g[sl].transpose(0, 2, 3, 1)), 1, 1, r["p"],
                      "x3", None, g_W, r["ws"])
        torch.cuda.synchronize()
        gWs.append(host(g_W))
    assert rel_l2(gWs[0], sum(gWs[1:])) <= 1e-5


# ---------------------------------------------------------------------------
# bf16 (the conv workloads' precision) against the oracle on bf16-rounded
# contraction operands (reading R9): s and W in the forward; dw^, s and W in
# the backward. Layer shapes, tau and M of configs 4 and 5 at a reduced image
# size (the oracle's contraction is a plain per-tap einsum), B = 2.
#
# The backward is compared at the GPU's own spike state (t, q, dv^/dt from
# the saved buffer), which the forward check has just held to the
# tolerance: the input-time gradient is a difference of dS at the two grid
# points around each input spike (for tau = (inf, inf) exactly (dS_{k+1} -
# dS_k) / dt), so it magnifies a spike-time difference by about T / dt, and
# bf16 operands legitimately move spike times by a few 1e-6. Likewise a
# dw^ entry at a bf16 rounding midpoint may round to either neighbour (fp32
# on the GPU, float64 in the oracle): the tolerance is 1e-3 plus that
# entry-wise bound (helpers.bf16_grad_rel_bound).
# ---------------------------------------------------------------------------
BF16_CASES = [
    # C_in, H, C_out, stride, tau, M
    (3, 16, 64, 1, (INF, INF), 32),       # config 4, layer 1
    (64, 16, 64, 2, (INF, INF), 32),      # config 4, layer 2
    (64, 8, 128, 1, (INF, INF), 32),      # config 4, layer 3
    (256, 4, 512, 1, (INF, INF), 32),     # config 4, layer 7
    (1, 12, 64, 1, (1.0, 0.25), 64),      # config 5, layer 1
    (64, 10, 64, 1, (1.0, 0.25), 64),     # config 5, layers 2-6
    (64, 10, 128, 2, (1.0, 0.25), 64),    # config 5, layer 7
    (128, 6, 128, 1, (1.0, 0.25), 64),    # config 5, layers 8-13
    (128, 6, 256, 2, (1.0, 0.25), 64),    # config 5, layer 14
    (256, 4, 256, 1, (1.0, 0.25), 64),    # config 5, layers 15-19
]
# other filter sizes at stride 2: an odd grid (stride classes of unequal
# size), 1x1 without padding (positions no tap reaches: zero gradient) and
# 5x5 with padding 2 (one, two or three tap rows per class)
BF16_KP_CASES = [c + (3, 1) for c in BF16_CASES] + [
    (64, 9, 64, 2, (1.0, 0.25), 64, 3, 1),
    (64, 8, 64, 2, (1.0, 0.25), 64, 1, 0),
    (64, 9, 128, 2, (INF, INF), 32, 5, 2),
]


def gpu_spike_state(r, B, O, Ho, Wo):
    """The GPU's spike state of a conv layer as an oracle context [B, O, Ho, Wo]."""
    from helpers import decode_saved
    q, _, vd = decode_saved(r["saved"].cpu().numpy(), B * Ho * Wo, O)
    tr = lambda a: np.asarray(a, float).reshape(B, Ho, Wo, O).transpose(0, 3, 1, 2)
    t = np.asarray(r["t"], float)
    return {"t": t, "q": tr(q).astype(int), "vdot": tr(vd), "fired": np.isfinite(t)}


@pytest.mark.parametrize("policy", [1, 2], ids=["generated", "tma"])
@pytest.mark.parametrize("C,H,O,stride,tau,M,k,pad", BF16_KP_CASES)
def test_conv_bf16_matches_rounded_oracle(C, H, O, stride, tau, M, k, pad, policy):
    """Both operand paths of the forward and dW (binned input generated in
    shared memory from the records, or written out and read through TMA)
    against the oracle on bf16-rounded operands."""
    from paper_2607_14672_gb300 import dstd
    prev = dstd.conv_set_operand_policy(policy)
    try:
        _conv_bf16_case(C, H, O, stride, tau, M, k, pad)
    finally:
        dstd.conv_set_operand_policy(prev)


def _conv_bf16_case(C, H, O, stride, tau, M, k, pad):
    from paper_2607_14672_gb300 import dstd
    from helpers import (bf16, bf16_ambiguous_ulp, bf16_grad_rel_bound, bf16_potential_bound, check_bf16_times,
                         conv_neurons, grid_of, kernel_max)
    B = 2
    t, L = conv_case(B, C, H, O, k, stride, pad, M, tau, seed=7 * C + H + O + k, wmean=WMEAN64[tau] * 64 / C * 9 / k ** 2,
                     gammas=(0.05, 0.01, 1e-3), silent=0.1, t_offset=0.3 * 1.2 / M)
    r = run_conv_fwd(t, L, "bf16")
    T, dt = grid_of(L)
    tv, ti = tau
    s = odstd.binning(t.reshape(B, -1), T, dt, tv, ti).reshape(B, M, C, H, H)
    what = onet.conv_what(bf16(s), bf16(L["W"]), stride, pad)
    _, _, Ho, Wo, _ = what.shape
    flat = odstd.solve(what.reshape(B, O * Ho * Wo, M), T, dt, tv, ti, 1.0)
    ctx = {k: flat[k].reshape(B, O, Ho, Wo) for k in ("t", "q", "vpeak", "vdot", "fired")}
    kmax = kernel_max(T, tv, ti)

    def bound(idx):
        b, o, y, x = np.unravel_index(idx, (B, O, Ho, Wo))
        nc = conv_neurons(t, L, list(zip(b, o, y, x)))
        return bf16_potential_bound(nc["s"], nc["w"], ctx["q"].ravel()[idx], ctx["t"].ravel()[idx], T, tv, ti,
                                    kmax)

    n_cmp, n_bound = check_bf16_times(r["t"], ctx, L, bound)
    assert n_cmp > 0.2 * r["t"].size
    assert n_bound <= 0.01 * r["t"].size

    # backward at the GPU's spike state: random upstream gradient on every
    # neuron (the penalty gradient T' is added on both sides from the GPU's times)
    gs = gpu_spike_state(r, B, O, Ho, Wo)
    nrm = 1.0 / (B * Ho * Wo)
    g = np.random.default_rng(C + O).normal(0.0, 1.0, gs["t"].shape)
    _, gT = olosses.temporal_penalty(gs["t"], 0.35, 0.8, 0.05, 0.01, nrm)
    g_t_in = torch.empty_like(r["t_in"])
    g_W = torch.empty_like(r["W"])
    dstd.conv_bwd(r["t_in"], r["W"], r["t_out"], r["saved"], dev(g.transpose(0, 2, 3, 1)), stride, pad, r["p"],
                  "bf16", g_t_in, g_W, r["ws"])
    torch.cuda.synchronize()
    assert dstd.device_status(clear=True) == 0
    fl = {k: gs[k].reshape(B, -1) for k in ("t", "q", "vdot", "fired")}
    gw = odstd.solve_backward(fl, (g + gT).reshape(B, -1), T, dt, tv, ti, 1.0).reshape(B, O, Ho, Wo, M)
    gW, gsum = onet.conv_what_adjoint(bf16(gw), bf16(s), bf16(L["W"]), stride, pad)
    ds = odstd.binning(t.reshape(B, -1), T, dt, tv, ti, derivative=True).reshape(gsum.shape)
    gin = np.sum(gsum * ds, axis=1)
    cnt = (~gs["fired"]).sum((0, 2, 3))
    gW = gW - 1e-3 * nrm * cnt[:, None, None, None]
    # dw^ entries at a bf16 rounding midpoint may round either way (bf16_grad_rel_bound)
    bW, bs = onet.conv_what_adjoint(bf16_ambiguous_ulp(gw, 2.0 ** -16), np.abs(bf16(s)), np.abs(bf16(L["W"])),
                                    stride, pad)
    b_in = np.sum(bs * np.abs(ds), axis=1)
    e_w = rel_l2(host(g_W).transpose(0, 3, 1, 2), gW)
    e_g = rel_l2(host(g_t_in).transpose(0, 3, 1, 2), gin)
    a_w, a_g = bf16_grad_rel_bound(bW, gW), bf16_grad_rel_bound(b_in, gin)
    assert e_w <= 1e-3 + a_w and e_g <= 1e-3 + a_g, (e_w, a_w, e_g, a_g)
    assert np.all(host(g_t_in).transpose(0, 3, 1, 2)[~np.isfinite(t)] == 0)


def test_conv_bf16_chunks_agree():
    """The implicit-GEMM path in chunks of whole images (1, 2 and 3 images
    per chunk, the last one ragged) against one chunk: the forward of an
    image does not depend on the chunk it falls in (bitwise), and dW sums
    the chunks' contributions (fp32 atomics: rounding order only)."""
    from paper_2607_14672_gb300 import dstd
    t, L = conv_case(5, 64, 10, 128, 3, 2, 1, 64, (1.0, 0.25), seed=21, wmean=WMEAN64[(1.0, 0.25)],
                     gammas=(0.05, 0.01, 1e-3), t_offset=0.005)
    outs = []
    prev = dstd.conv_set_chunk_images(0)
    try:
        for cap in (0, 1, 2, 3):
            dstd.conv_set_chunk_images(cap)
            r = run_conv_fwd(t, L, "bf16")
            g = np.where(np.isfinite(r["t"]), 1.0, 0.0)
            g_t_in = torch.empty_like(r["t_in"])
            g_W = torch.empty_like(r["W"])
            dstd.conv_bwd(r["t_in"], r["W"], r["t_out"], r["saved"], dev(g.transpose(0, 2, 3, 1)), 2, 1, r["p"],
                          "bf16", g_t_in, g_W, r["ws"])
            torch.cuda.synchronize()
            assert dstd.device_status(clear=True) == 0
            outs.append((r["t"], host(g_t_in), host(g_W)))
    finally:
        dstd.conv_set_chunk_images(prev)
    t0, gi0, gw0 = outs[0]
    assert np.isfinite(t0).mean() > 0.2
    for tt, gi, gw in outs[1:]:
        np.testing.assert_array_equal(tt, t0)
        assert rel_l2(gi, gi0) <= 1e-6
        assert rel_l2(gw, gw0) <= 1e-5
