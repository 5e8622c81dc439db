"""GPU parity of the multi-spike layer (App. D) against the float64 oracle
(``oracle/multispike.py``), three-product mode (fp32 accuracy).

Every spike time of every neuron is compared (1e-4 T_max), and the spike
counts exactly, except for neurons whose potential came within 1e-5 of the
threshold in an interval that decided a spike (the oracle's ``margin``).
Gradients (dW and the input-time gradient of every input spike) within 1e-3
relative L2, with the upstream gradient of those near-threshold neurons set
to zero on both sides.
"""

import math

import numpy as np
import pytest
import torch

from helpers import f32, grid_of, rel_l2
from oracle import multispike as oms

pytestmark = pytest.mark.gpu

INF = math.inf
TAUS = [(0.5, 0.25), (INF, INF), (INF, 0.3), (0.3, INF), (0.4, 0.4), (1.0, 0.25)]


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2607_14672_gb300 import build, dstd
    build.build()
    dstd.load()
    assert dstd.device_status(clear=True) == 0
    yield
    assert dstd.device_status(clear=True) == 0


def layer(seed, B, N_in, N_out, F_in, tau_v, tau_I, M=16):
    g = np.random.default_rng(seed)
    t = np.sort(g.uniform(0.0, 1.0, (B, N_in, F_in)), axis=-1)
    t[g.random(t.shape) < 0.25] = INF
    t = np.sort(t, axis=-1)
    # a mean that makes most neurons fire several times in the window
    scale = {(INF, INF): 2.5, (INF, 0.3): 4.0, (0.3, INF): 4.0}.get((tau_v, tau_I), 6.0)
    W = g.normal(scale / (N_in * F_in * 0.75) * 4.0, 1.5 / math.sqrt(N_in), (N_out, N_in))
    L = dict(tau_v=tau_v, tau_I=tau_I, v_th=1.0, t_first=0.0, t_end=1.2, M=M, t_offset=0.011)
    return f32(t), f32(W), L


def run(t, W, L, F_out, g_up=None, math_mode="x3"):
    from paper_2607_14672_gb300 import dstd
    B, N_in, F_in = t.shape
    N_out = W.shape[0]
    p = dstd.params(dict(L, t_head_l=0.0, t_tail_l=0.0), 0.0)
    ws = torch.empty(dstd.ms_workspace_bytes(B, N_in, N_out, F_in, F_out, p, math_mode), dtype=torch.uint8,
                     device="cuda")
    saved = torch.empty(dstd.ms_saved_bytes(B, N_out, F_out), dtype=torch.uint8, device="cuda")
    t_in = torch.tensor(t, dtype=torch.float32, device="cuda")
    Wd = torch.tensor(W, dtype=torch.float32, device="cuda")
    t_out = torch.empty(B, N_out, F_out, device="cuda")
    dstd.dense_fwd_ms(t_in, Wd, p, math_mode, t_out, saved, ws)
    out = {"t": t_out.cpu().numpy().astype(np.float64)}
    if g_up is not None:
        g_in = torch.empty_like(t_in)
        g_W = torch.empty_like(Wd)
        dstd.dense_bwd_ms(t_in, Wd, t_out, saved, torch.tensor(g_up, dtype=torch.float32, device="cuda"), p,
                          math_mode, g_in, g_W, ws)
        out["g_in"] = g_in.cpu().numpy().astype(np.float64)
        out["g_W"] = g_W.cpu().numpy().astype(np.float64)
    torch.cuda.synchronize()
    assert dstd.device_status(clear=True) == 0
    return out


def compare_times(tg, ctx, L, margin=1e-5):
    ok = ctx["margin"] > margin
    ng, no = np.isfinite(tg).sum(-1), np.isfinite(ctx["t"]).sum(-1)
    assert not (ok & (ng != no)).any(), int((ok & (ng != no)).sum())
    both = ok[..., None] & np.isfinite(tg) & np.isfinite(ctx["t"])
    assert both.any()
    assert np.abs(tg[both] - ctx["t"][both]).max() <= 1e-4 * (L["t_end"] - L["t_first"])
    return ok, no


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
@pytest.mark.parametrize("shape", [(4, 40, 24, 3, 4), (3, 130, 150, 2, 3), (2, 7, 5, 1, 6)])
def test_multispike_forward_matches_oracle(tau_v, tau_I, shape):
    B, N_in, N_out, F_in, F_out = shape
    t, W, L = layer(N_in + 7 * N_out, B, N_in, N_out, F_in, tau_v, tau_I)
    T, dt = grid_of(L)
    ctx = oms.dstd_forward_ms(t, W, T, dt, tau_v, tau_I, 1.0, F_out)
    g = run(t, W, L, F_out)
    ok, n = compare_times(g["t"], ctx, L)
    assert (n >= 2).sum() >= max(2, n.size // 20)          # the reset path is exercised
    # ascending, inside the window, +inf after the last spike
    tg = g["t"]
    fin = np.isfinite(tg)
    assert np.all(np.diff(np.where(fin, tg, 1e9), axis=-1) >= 0)
    assert np.all(tg[fin] < L["t_end"])


@pytest.mark.parametrize("tau_v,tau_I", [(0.5, 0.25), (INF, INF), (INF, 0.3), (1.0, 0.25)])
def test_multispike_backward_matches_oracle(tau_v, tau_I):
    B, N_in, N_out, F_in, F_out = 4, 60, 40, 2, 4
    t, W, L = layer(5, B, N_in, N_out, F_in, tau_v, tau_I)
    T, dt = grid_of(L)
    ctx = oms.dstd_forward_ms(t, W, T, dt, tau_v, tau_I, 1.0, F_out)
    ok = ctx["margin"] > 1e-4
    up = np.random.default_rng(3).normal(size=ctx["t"].shape)
    up = np.where(ok[..., None] & np.isfinite(ctx["t"]), up, 0.0)
    g = run(t, W, L, F_out, g_up=up.astype(np.float32))
    compare_times(g["t"], ctx, L)
    gW, gin, _ = oms.dstd_backward_ms(ctx, t, W, up, T, dt, tau_v, tau_I, 1.0)
    assert (np.isfinite(ctx["t"]).sum(-1) >= 2).sum() >= 10
    assert rel_l2(g["g_W"], gW) <= 1e-3
    gin = np.where(np.isfinite(t), gin, 0.0)
    assert rel_l2(g["g_in"], gin) <= 1e-3


def test_multispike_single_spike_equals_ttfs_layer():
    # F_in = F_out = 1: the same spikes as the first-spike layer
    from paper_2607_14672_gb300 import dstd
    t, W, L = layer(9, 4, 64, 48, 1, 0.5, 0.25)
    g = run(t, W, L, 1)
    p = dstd.params(dict(L, t_head_l=0.0, t_tail_l=0.0), 0.0)
    ws = torch.empty(dstd.dense_workspace_bytes(4, 64, 48, p, "x3"), dtype=torch.uint8, device="cuda")
    t_out = torch.empty(4, 48, device="cuda")
    saved = torch.empty(dstd.dense_saved_bytes(4, 48), dtype=torch.uint8, device="cuda")
    pen = torch.empty(4, device="cuda")
    dstd.dense_fwd(torch.tensor(t[..., 0], dtype=torch.float32, device="cuda"),
                   torch.tensor(W, dtype=torch.float32, device="cuda"), p, "x3", t_out, saved, pen, ws)
    ref = t_out.cpu().numpy().astype(np.float64)
    a = g["t"][..., 0]
    np.testing.assert_array_equal(np.isfinite(a), np.isfinite(ref))
    fin = np.isfinite(a)
    assert np.abs(a[fin] - ref[fin]).max() <= 1e-5


def test_multispike_arguments_rejected():
    from paper_2607_14672_gb300 import dstd
    t, W, L = layer(1, 2, 8, 4, 2, 0.5, 0.25)
    p = dstd.params(dict(L, t_head_l=0.0, t_tail_l=0.0), 0.0)
    assert dstd.ms_workspace_bytes(2, 8, 4, 9, 2, p, "x3") == 0          # F_in above 8
    assert dstd.ms_workspace_bytes(2, 8, 4, 2, 2, p, "f32") == 0         # CUDA-core mode unsupported
    assert dstd.ms_saved_bytes(2, 4, 0) == 0
