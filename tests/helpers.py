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


# ---------------------------------------------------------------------------
# bf16 operands (reading R9): which differences from the oracle are legitimate
# ---------------------------------------------------------------------------
def bf16_ulp(x):
    """Spacing of bfloat16 numbers (8 significant bits) at |x|."""
    a = np.abs(np.asarray(x, float))
    safe = np.where((a > 0) & np.isfinite(a), a, 1.0)
    return np.where((a > 0) & np.isfinite(a), 2.0 ** (np.floor(np.log2(safe)) - 7), 0.0)


def bf16_ambiguous_ulp(x, rel=2.0 ** -18):
    """One bf16 step where x lies within ``rel`` |x| of a rounding midpoint, else 0.

    The CUDA path rounds a grid weight to bf16 from its fp32 value, the oracle
    from its float64 value; the two differ by a few fp32 ulps (2^-18 is 64 of
    them), so only weights this close to a midpoint can round to different
    bf16 neighbours, by one step.
    """
    a = np.abs(np.asarray(x, float))
    u = bf16_ulp(a)
    f = np.where(u > 0, a / np.where(u > 0, u, 1.0), 0.0)
    amb = (u > 0) & (np.abs(f - np.floor(f) - 0.5) * u <= rel * a)
    return np.where(amb, u, 0.0)


def bf16_potential_bound(s, w, q, t, T, tau_v, tau_I, kmax, v_th=1.0):
    """Bound on |v^_gpu - v^_oracle| of bf16-operand neurons.

    s [n, M, K] grid weights (float64, unrounded), w [n, K] weights, q [n]
    spike interval (M when silent), t [n] oracle spike time. Per grid point:
    (1) grid weights that may round to the other bf16 neighbour
    (``bf16_ambiguous_ulp``); (2) the fp32 accumulation of the exact bf16 x
    bf16 products, at most (nnz - 1) 2^-23 sum |terms| with nnz nonzero
    terms (the recursive-summation bound; 2^-23 allows truncating adds);
    (3) the fp32 scan of the state over at most M grid steps, four roundings
    each: M 2^-22 sum |terms|. At the spike, also the root's stopping
    tolerance, |v^ - v_th| <= 4e-7 v_th. Returns (bound at the spike, bound
    over the whole window).
    """
    from oracle import lif
    aw = np.abs(np.asarray(w, float))[:, None, :]
    amb = np.sum(bf16_ambiguous_ulp(s) * aw, -1)                          # [n, M]
    terms = np.abs(bf16(s)) * aw
    nnz = np.count_nonzero(terms, -1)
    M = s.shape[1]
    arith = (2.0 ** -23 * np.maximum(nnz - 1, 0) + M * 2.0 ** -22) * terms.sum(-1)
    per_m = amb + arith
    fired = q < M
    ts = np.where(fired, t, T[0])
    Km = lif.K(ts[:, None] - T[None, :M], tau_v, tau_I)
    upto = np.arange(M)[None, :] <= np.minimum(q, M - 1)[:, None]
    at_spike = np.sum(np.where(upto & fired[:, None], per_m * Km, 0.0), -1) + 4e-7 * v_th
    return at_spike, kmax * per_m.sum(-1)


def kernel_max(T, tau_v, tau_I):
    """max of K(s) over the window (K >= 0, single hump or monotone)."""
    from oracle import lif
    s = np.linspace(0.0, T[-1] - T[0], 20001)
    return float(lif.K(s, tau_v, tau_I).max()) * (1.0 + 1e-6)


def check_bf16_times(t_gpu, ctx, layer, bound_fn, base=1e-4, margin=1e-5):
    """Spike times and masks of a bf16 layer against the oracle on bf16-rounded operands.

    Every neuron must meet the benchmark spec's tolerance (|dt| <= base T_max; masks
    equal where the peak potential is more than ``margin`` from the
    threshold), widened only by the neuron's own potential bound
    (``bound_fn(flat indices) -> (at spike, whole window)``, usually
    ``bf16_potential_bound``), divided by dv^/dt at the spike for the time.
    Returns (neurons compared, neurons that needed their bound).
    """
    Tmax = layer["t_end"] - layer["t_first"]
    t_gpu = np.asarray(t_gpu, float).ravel()
    t_o = np.asarray(ctx["t"], float).ravel()
    vpeak = np.asarray(ctx["vpeak"], float).ravel()
    vdot = np.asarray(ctx["vdot"], float).ravel()
    fo, fg = np.isfinite(t_o), np.isfinite(t_gpu)
    far = np.abs(vpeak - layer["v_th"]) > margin
    both = far & fo & fg
    err = np.where(both, np.abs(np.where(both, t_gpu, 0.0) - np.where(both, t_o, 0.0)), 0.0)
    flag = (far & (fo != fg)) | (err > base * Tmax)
    idx = np.flatnonzero(flag)
    if idx.size:
        dv_spike, dv_all = bound_fn(idx)
        flips = fo[idx] != fg[idx]
        assert np.all(~flips | (np.abs(vpeak[idx] - layer["v_th"]) <= margin + dv_all)), \
            f"{int(np.sum(flips & (np.abs(vpeak[idx] - layer['v_th']) > margin + dv_all)))} mask flips beyond the bound"
        floor = 1e-6 * layer["v_th"] / ((layer["t_end"] - layer["t_first"]) / layer["M"])
        allowed = base * Tmax + dv_spike / np.maximum(np.where(np.isfinite(vdot[idx]), vdot[idx], floor), floor)
        tb = ~flips
        assert np.all(err[idx][tb] <= allowed[tb]), \
            f"max |dt| / allowed = {np.max(err[idx][tb] / allowed[tb]):.3f}"
    return int(both.sum()), int(idx.size)


# ---------------------------------------------------------------------------
# conv neurons computed one by one from their receptive fields (oracle steps)
# ---------------------------------------------------------------------------
def receptive_fields(x, k, stride, pad, pos):
    """Spike times under the k x k filter of output positions pos = [(b, y, x)]
    of a conv over x [B, C, H, W] with silent padding: [n, C * k * k] in
    (c, kh, kw) order (the oracle's filter order)."""
    xp = np.pad(np.asarray(x, float), ((0, 0), (0, 0), (pad, pad), (pad, pad)), constant_values=np.inf)
    return np.stack([xp[b, :, y * stride:y * stride + k, xx * stride:xx * stride + k].reshape(-1)
                     for (b, y, xx) in pos])


def conv_neurons(x, layer, neurons, operand_round=bf16):
    """Oracle forward of conv neurons [(b, o, y, x)] from their receptive fields
    on rounded contraction operands. Returns the ``solve`` dict plus s [n, M, K]
    (unrounded grid weights) and w [n, K]."""
    T, dt = grid_of(layer)
    W = np.asarray(layer["W"], np.float32).astype(np.float64)
    O, C, k, _ = W.shape
    rf = receptive_fields(x, k, layer["stride"], layer["pad"], [(b, y, xx) for (b, _, y, xx) in neurons])
    s = odstd.binning(rf, T, dt, layer["tau_v"], layer["tau_I"])          # [n, M, K]
    w = W.reshape(O, -1)[[o for (_, o, _, _) in neurons]]
    what = np.einsum("nmj,nj->nm", operand_round(s), operand_round(w))
    ctx = odstd.solve(what[None], T, dt, layer["tau_v"], layer["tau_I"], layer["v_th"])
    ctx = {key: ctx[key][0] for key in ("t", "q", "vpeak", "vdot", "fired")}
    ctx.update(s=s, w=w, T=T, dt=dt, what=what)
    return ctx


def neuron_bound_fn(ctx, layer):
    """bound_fn for ``check_bf16_times`` over neurons whose ctx holds s [n, M, K] and w [n, K]."""
    T = ctx["T"]
    kmax = kernel_max(T, layer["tau_v"], layer["tau_I"])

    def fn(idx):
        return bf16_potential_bound(ctx["s"][idx], ctx["w"][idx], np.asarray(ctx["q"]).ravel()[idx],
                                    np.asarray(ctx["t"]).ravel()[idx], T, layer["tau_v"], layer["tau_I"], kmax)
    return fn


def dense_bound_fn(ctx, W, layer):
    """bound_fn for a dense layer's ctx from ``oracle_forward`` (s [B, M, N_in])."""
    T = ctx["T"]
    kmax = kernel_max(T, layer["tau_v"], layer["tau_I"])
    W = np.asarray(W, float)
    shape = np.asarray(ctx["t"]).shape

    def fn(idx):
        b, i = np.unravel_index(idx, shape)
        return bf16_potential_bound(ctx["s"][b], W[i], ctx["q"][b, i], ctx["t"][b, i], T, layer["tau_v"],
                                    layer["tau_I"], kmax)
    return fn


def bf16_grad_rel_bound(bound, ref):
    """The relative L2 allowance a bf16 backward adds to the benchmark spec's 1e-3:
    ||per-element bound|| / ||reference||. The per-element bound sums, over
    the dC/dw^ entries that lie within 2^-16 of a bf16 rounding midpoint (the
    GPU rounds its fp32 value, the oracle its float64 one: they may land on
    different neighbours), one bf16 step times the other operand's
    magnitude (and |ds/dt| for the input-time gradient)."""
    n = np.linalg.norm(np.asarray(ref, float))
    return float(np.linalg.norm(np.asarray(bound, float)) / n) if n > 0 else 0.0
