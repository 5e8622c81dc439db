"""Shared helpers of the parity tests (test code only)."""

import numpy as np

from oracle import dstd as odstd

INF = np.inf


def f32(x):
    """Round to float32 and back: the inputs exactly as the CUDA path sees them."""
    return np.asarray(x, np.float32).astype(np.float64)


def bf16(x):
    """Round-to-nearest-even to bfloat16 (8 significant bits), as float64."""
    a = np.ascontiguousarray(np.asarray(x, np.float32))
    u = a.view(np.uint32).astype(np.uint64)
    rounding = ((u >> 16) & 1) + 0x7FFF
    r = ((u + rounding) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32).astype(np.float64)
    return np.where(np.isfinite(a), out, a.astype(np.float64))


def grid_of(layer):
    return odstd.grid(layer["t_first"], layer["t_end"], layer["M"], layer.get("t_offset", 0.0))


def oracle_forward(t_in, W, layer, solver="table", operand_round=None):
    """Oracle DSTD forward of one dense layer; ``operand_round`` (e.g. bf16)
    rounds the two contraction operands s and W first."""
    T, dt = grid_of(layer)
    tv, ti, V = layer["tau_v"], layer["tau_I"], layer["v_th"]
    if operand_round is None:
        ctx = odstd.forward_dense(t_in, W, T, dt, tv, ti, V, solver)
    else:
        s = odstd.binning(t_in, T, dt, tv, ti)
        what = np.einsum("bmj,ij->bim", operand_round(s), operand_round(W))
        ctx = odstd.solve(what, T, dt, tv, ti, V, solver)
        ctx.update(s=s, what=what)
    ctx["T"], ctx["dt"] = T, dt
    return ctx


def decode_saved(raw, B, N):
    """Split the opaque saved buffer into (q, s, vdot) [B, N] (256-byte aligned arrays)."""
    raw = np.asarray(raw, np.uint8)
    n = B * N * 4
    o1 = (n + 255) // 256 * 256
    o2 = (o1 + n + 255) // 256 * 256
    q = raw[:n].view(np.int32).reshape(B, N)
    s = raw[o1:o1 + n].view(np.float32).reshape(B, N)
    vd = raw[o2:o2 + n].view(np.float32).reshape(B, N)
    return q, s, vd


def well_conditioned(ctx, v_th, margin=1e-5):
    """Neurons whose peak potential is not within ``margin`` of the threshold."""
    return np.abs(ctx["vpeak"] - v_th) > margin


def rel_l2(a, b):
    a = np.asarray(a, float)
    b = np.asarray(b, float)
    d = np.linalg.norm(a - b)
    n = np.linalg.norm(b)
    return d / n if n > 0 else d


def dense_layer(B, N_in, N_out, M, tau_v, tau_I, seed=0, fire=0.5, wstd_scale=1.0, t_first=0.0, t_end=1.2,
                t_offset=0.0, silent=0.2, t_hi=1.0, gammas=(0.0, 0.0, 0.0), edges=(0.3, 0.9)):
    """A random dense layer dict and inputs for parity tests.

    Inputs U[0, t_hi) with a ``silent`` share; W = mu + N(0, wstd_scale^2/N_in)
    with mu found by oracle bisection so that about ``fire`` of the neurons
    fire on the first (up to) 8 samples.
    """
    from paper_2607_14672_gb300 import synth
    t_in = synth.uniform_spikes(seed, (B, N_in), 0.0, t_hi, silent)
    Z = synth.normal_weights(seed + 1000, (N_out, N_in), 0.0, wstd_scale / np.sqrt(N_in))
    layer = dict(kind="dense", W=None, tau_v=tau_v, tau_I=tau_I, v_th=1.0, M=M, t_first=t_first, t_end=t_end,
                 t_offset=t_offset, t_head_l=edges[0], t_tail_l=edges[1], gamma_head=gammas[0],
                 gamma_tail=gammas[1], gamma_q=gammas[2])
    T, dt = grid_of(layer)
    sub = f32(t_in[:8])
    Zs = Z[:64]
    lo, hi = 0.0, 1.0
    while np.isfinite(odstd.forward_dense(sub, Zs + hi, T, dt, tau_v, tau_I, 1.0)["t"]).mean() < fire and hi < 1e6:
        lo, hi = hi, hi * 2
    for _ in range(24):
        mid = 0.5 * (lo + hi)
        f = np.isfinite(odstd.forward_dense(sub, Zs + mid, T, dt, tau_v, tau_I, 1.0)["t"]).mean()
        lo, hi = (mid, hi) if f < fire else (lo, mid)
    layer["W"] = Z + hi
    return t_in, layer
