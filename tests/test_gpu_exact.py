"""GPU exact (event-driven) forward, Alg. 1, against the oracle's exact method.

The oracle sorts each sample's inputs and solves every inter-spike interval
with the closed forms of Tab. spike_timing (or its bracketed solver); the GPU
walks the same intervals with the decayed (v, I) state. Spike times must agree
within 1e-4 T_max and the firing masks exactly, except for neurons whose peak
potential comes within 1e-5 of the threshold (found with the oracle's own
per-interval maxima).
"""

import numpy as np
import pytest
import torch

from helpers import dense_layer, f32
from oracle import exact as oexact, lif

pytestmark = pytest.mark.gpu

INF = float("inf")
TAUS = [(0.5, 0.25), (INF, INF), (INF, 0.3), (0.3, INF), (0.4, 0.4), (1.0, 0.25), (0.25, 0.5)]


def dev(x):
    return torch.tensor(np.asarray(x, np.float32), device="cuda")


def exact_peak(t_in, W, tau_v, tau_I, t_end):
    """Peak potential of every neuron over [first input, t_end) (oracle)."""
    case = lif.lif_case(tau_v, tau_I)
    out = np.full((t_in.shape[0], W.shape[0]), -np.inf)
    for b in range(t_in.shape[0]):
        fin = np.isfinite(t_in[b]) & (t_in[b] < t_end)
        if not fin.any():
            continue
        order = np.argsort(t_in[b][fin], kind="stable")
        tt = t_in[b][fin][order]
        Wt = W[:, fin][:, order].astype(float)
        lo = tt
        hi = np.minimum(np.append(tt[1:], np.inf), t_end)
        c = lif.interval_coeffs(case, tau_v, tau_I, np.broadcast_to(tt, Wt.shape), Wt, tt[0])
        out[b] = lif.interval_peak(c, np.broadcast_to(lo, Wt.shape), np.broadcast_to(hi, Wt.shape)).max(-1)
    return out


def run_exact(t_in, layer):
    from paper_2607_14672_gb300 import dstd
    B, N_in = t_in.shape
    N_out = layer["W"].shape[0]
    p = dstd.params(layer, 1.0 / B)
    ws = torch.empty(dstd.exact_workspace_bytes(B, N_in, N_out), dtype=torch.uint8, device="cuda")
    t_out = torch.empty(B, N_out, device="cuda")
    dstd.exact_fwd(dev(t_in), dev(layer["W"]), p, t_out, ws)
    torch.cuda.synchronize()
    assert dstd.device_status(clear=True) == 0
    return t_out.cpu().numpy()


@pytest.mark.parametrize("tau_v,tau_I", TAUS)
@pytest.mark.parametrize("shape", [(6, 37, 50), (4, 300, 129), (3, 1, 5), (2, 1000, 40)])
def test_exact_forward_matches_oracle(tau_v, tau_I, shape):
    B, N_in, N_out = shape
    t_in, layer = dense_layer(B, N_in, N_out, 32, tau_v, tau_I, seed=N_in + N_out, fire=0.6)
    t_in, layer["W"] = f32(t_in), f32(layer["W"])
    t_end = layer["t_end"]
    t_gpu = run_exact(t_in, layer)
    t_ref = oexact.exact_forward(t_in, layer["W"], tau_v, tau_I, layer["v_th"], t_end=t_end)
    ok = np.abs(exact_peak(t_in, layer["W"], tau_v, tau_I, t_end) - layer["v_th"]) > 1e-5
    fin_g, fin_r = np.isfinite(t_gpu), np.isfinite(t_ref)
    assert not (ok & (fin_g != fin_r)).any()
    both = ok & fin_g & fin_r
    Tmax = layer["t_end"] - layer["t_first"]
    if both.any():
        assert np.abs(t_gpu[both] - t_ref[both]).max() <= 1e-4 * Tmax
    # spikes lie inside the window, after the sample's first input
    first = np.where(np.isfinite(t_in), t_in, np.inf).min(1, keepdims=True)
    assert np.all(t_gpu[fin_g] < t_end) and np.all((t_gpu >= first)[fin_g])


def test_exact_forward_edge_cases():
    """All inputs silent, all after the window, and a single input spike with
    a weight that crosses the threshold (closed form of Tab. spike_timing for
    tau_v = inf: v = w (1 - e^{-t/tau_s}) tau_s)."""
    t_in, layer = dense_layer(3, 16, 8, 32, INF, 0.25, seed=3, fire=0.5)
    t_in = np.full_like(f32(t_in), np.inf)
    t_in[1, :] = 5.0                      # after the window end (1.2)
    t_in[2, :] = np.inf
    t_in[2, 3] = 0.1
    W = np.zeros((8, 16), np.float32)
    W[:, 3] = np.linspace(1.0, 12.0, 8)   # v(t) -> w tau_s: fires when w tau_s > v_th
    layer["W"] = W
    t = run_exact(t_in, layer)
    assert np.isinf(t[0]).all() and np.isinf(t[1]).all()
    w = W[:, 3].astype(float)
    with np.errstate(divide="ignore", invalid="ignore"):
        s = -0.25 * np.log1p(-1.0 / (w * 0.25))        # w tau_s (1 - e^{-s/tau_s}) = 1
    expect = np.where(w * 0.25 > 1.0, 0.1 + s, np.inf)
    expect = np.where(expect < layer["t_end"], expect, np.inf)
    fin = np.isfinite(expect)
    assert (np.isfinite(t[2]) == fin).all()
    assert np.abs(t[2][fin] - expect[fin]).max() <= 1e-5


@pytest.mark.parametrize("tau_v,tau_I", [(0.5, 0.25), (INF, INF), (0.4, 0.4), (1.0, 0.25), (INF, 0.3)])
@pytest.mark.parametrize("shape", [(6, 37, 50), (4, 300, 129), (2, 1000, 40)])
def test_exact_backward_matches_oracle(tau_v, tau_I, shape):
    """The exact backward on the GPU against oracle.exact.exact_backward at
    the GPU's own spike times (float64 on the oracle side): g_W and g_t_in
    within 1e-4 relative L2. Neurons whose slope at the crossing is under a
    twentieth of the median get no upstream gradient (1/V' would magnify
    fp32 rounding there)."""
    from paper_2607_14672_gb300 import dstd
    B, N_in, N_out = shape
    t_in, layer = dense_layer(B, N_in, N_out, 32, tau_v, tau_I, seed=N_in + 2 * N_out, fire=0.6)
    t_in, W = f32(t_in), f32(layer["W"])
    layer["W"] = W
    t_out = run_exact(t_in, layer)
    fired = np.isfinite(t_out)
    assert fired.sum() > 0.2 * t_out.size
    # slope at each spike (oracle), to leave out near-tangential crossings
    x = np.where(fired[:, :, None], t_out[:, :, None], 0.0) - np.where(np.isfinite(t_in), t_in, INF)[:, None, :]
    causal = fired[:, :, None] & np.isfinite(t_in)[:, None, :] & (x > 0)
    Vp = np.einsum("bij,ij->bi", np.where(causal, lif.K_prime(np.where(causal, x, 0.0), tau_v, tau_I), 0.0),
                   W.astype(float))
    g = np.random.default_rng(N_in).normal(0.0, 1.0, t_out.shape)
    g = np.where(fired & (Vp > 0.05 * np.median(Vp[fired])), g, 0.0)
    gW_ref, gT_ref = oexact.exact_backward(t_in, W, t_out, g, tau_v, tau_I)
    p = dstd.params(layer, 1.0 / B)
    ws = torch.empty(dstd.exact_workspace_bytes(B, N_in, N_out), dtype=torch.uint8, device="cuda")
    gW = torch.empty(N_out, N_in, device="cuda")
    gT = torch.empty(B, N_in, device="cuda")
    dstd.exact_bwd(dev(t_in), dev(W), dev(t_out), dev(g), p, gT, gW, ws)
    torch.cuda.synchronize()
    assert dstd.device_status(clear=True) == 0
    rel = lambda a, b: np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30)
    assert rel(gW.cpu().numpy(), gW_ref) <= 1e-4, rel(gW.cpu().numpy(), gW_ref)
    assert rel(gT.cpu().numpy(), gT_ref) <= 1e-4, rel(gT.cpu().numpy(), gT_ref)
    # without g_t_in only g_W is written
    gW2 = torch.full((N_out, N_in), float("nan"), device="cuda")
    dstd.exact_bwd(dev(t_in), dev(W), dev(t_out), dev(g), p, None, gW2, ws)
    torch.cuda.synchronize()
    assert torch.equal(gW2, gW)
