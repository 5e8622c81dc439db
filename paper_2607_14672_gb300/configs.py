"""Workload definitions: shapes, constants, seeds (no arithmetic of the method).

Every workload is synthetic and seeded (``synth``); the image datasets of the
paper's experiments are replaced by inputs of the same shape and value range.
A layer is a plain dict understood by both the CUDA driver (``net.py``) and
the float64 oracle:

  kind            "dense" | "conv"
  W               float64 weights, dense [N_out, N_in], conv [C_out, C_in, k, k]
  tau_v, tau_I    membrane / synaptic time constants (math.inf allowed)
  v_th            threshold
  t_first, t_end  DSTD window; M steps; grid T_m = t_first + m dt - t_offset
  t_offset        in (-dt/2, dt/2]
  t_head_l, t_tail_l, gamma_head, gamma_tail, gamma_q  synfire penalty terms
  conv only       stride, pad, in_shape (C, H, W)

Synfire constants follow App. C.1 with mid-range values of Tab. search_space:
tau_width = 1, tau_shift = 0.1, tau_margin = 0.1, t_head = t_tail = 0.2,
gamma_head = 0.05, gamma_tail = 0.01, gamma_Q = 1e-3, tau_soft = 0.02, tau_in = 1.
Layer l's window is [l tau_shift - tau_margin, l tau_shift + tau_width + tau_margin]
and its penalty edges t_head^(l) = l tau_shift + t_head,
t_tail^(l) = l tau_shift + tau_width - t_tail.

Weight means mu_l (configs 2-5, Syn-SNN-9/20) make about 80% of each layer's neurons fire
at initialisation on the seed-0 batch with t_offset = 0; they were found once
by bisection with the oracle (``oracle/calibrate_configs.py``) and are frozen
here.
"""

import math

import numpy as np

from . import synth

INF = math.inf

SYNFIRE = dict(tau_in=1.0, tau_width=1.0, tau_shift=0.1, tau_margin=0.1, t_head=0.2, t_tail=0.2,
               gamma_head=0.05, gamma_tail=0.01, gamma_q=1e-3, tau_soft=0.02)

# seeds: inputs 0, layer-l weights 1000 + l, labels 7, t_offset draws 11
SEED_INPUT, SEED_W, SEED_LABELS, SEED_OFFSET = 0, 1000, 7, 11

# frozen calibration (80% firing at init), see module docstring
CFG2_MU = (0.03523, 0.01520, 0.01951)
CFG3_MU_TIMES_N = 17.4
CFG4_MU = (0.09306, 0.00761, 0.01274, 0.01387, 0.00942, 0.00637, 0.00514, 0.00285, 0.00093)
SYN9_MU = (0.04479, 0.00758, 0.0125, 0.02298, 0.02083, 0.01099, 0.01407, 0.00318, 0.00084)
SYN20_MU = (0.28323, 0.00786, 0.01288, 0.00507, 0.01689, 0.02131, 0.00956, 0.00937, 0.01019, 0.00484, 0.01054,
            0.0105, 0.00636, 0.00449, 0.00506, 0.0024, 0.00522, 0.00541, 0.004, 0.00077)
CFG5_MU = (0.96918, 0.01896, 0.02438, 0.0258, 0.02676, 0.02719, 0.02923, 0.01346, 0.01353, 0.01343,
           0.01367, 0.01382, 0.01358, 0.01714, 0.00673, 0.00686, 0.00689, 0.00699, 0.00697, 0.00077)


def synfire_layer(l, syn=SYNFIRE):
    """Window and penalty edges of layer l >= 1 (App. C.1)."""
    return dict(
        t_first=l * syn["tau_shift"] - syn["tau_margin"],
        t_end=l * syn["tau_shift"] + syn["tau_width"] + syn["tau_margin"],
        t_head_l=l * syn["tau_shift"] + syn["t_head"],
        t_tail_l=l * syn["tau_shift"] + syn["tau_width"] - syn["t_tail"],
        gamma_head=syn["gamma_head"], gamma_tail=syn["gamma_tail"], gamma_q=syn["gamma_q"])


def _dense(W, tau_v, tau_I, M, t_first, t_end, v_th=1.0, **kw):
    d = dict(kind="dense", W=W, tau_v=tau_v, tau_I=tau_I, v_th=v_th, M=M, t_first=t_first,
             t_end=t_end, t_offset=0.0, t_head_l=0.0, t_tail_l=0.0, gamma_head=0.0,
             gamma_tail=0.0, gamma_q=0.0)
    d.update(kw)
    return d


def config1(scale=1.0, batch=8):
    """Single dense layer 64 -> 32, B = 8, M = 16 over [0, 1], (tau_m, tau_s) = (0.5, 0.25).

    Inputs U[0, 0.8) with 20% silent; W ~ N(0, 1/64) * 4 * scale (scale 12 is
    the "1b" variant, where about a third of the outputs fire); loss = sum of
    the output spike times that fire.
    """
    W = synth.normal_weights(SEED_W + 1, (32, 64), 0.0, 1.0 / 8.0) * 4.0 * scale
    return dict(
        name="cfg1" if scale == 1.0 else "cfg1b",
        workload=f"dense LIF layer 64->32, B={batch}, M=16, tau=(0.5,0.25)" + ("" if scale == 1.0 else " x12 weights"),
        batch=batch, in_shape=(64,), loss="sum_t", tau_soft=None,
        inputs=lambda seed=SEED_INPUT, B=batch: synth.uniform_spikes(seed, (B, 64), 0.0, 0.8, 0.2),
        layers=[_dense(W, 0.5, 0.25, 16, 0.0, 1.0)])


def config2(batch=256, M=32):
    """3-layer dense MLP 784-800-800-10, B = 256, M = 32, (tau_m, tau_s) = (0.5, 0.25).

    Inputs: 28x28 intensities x ~ U[0,1) with 60% zeros, t = 1 - x (x = 0
    silent); synfire windows per layer; loss = CE over softmax(-t/tau_soft)
    with 10 random labels + T + gamma_Q Q.
    """
    sizes = [784, 800, 800, 10]
    layers = []
    for l in range(1, 4):
        W = synth.normal_weights(SEED_W + l, (sizes[l], sizes[l - 1]), CFG2_MU[l - 1],
                                 1.0 / math.sqrt(sizes[l - 1]))
        layers.append(_dense(W, 0.5, 0.25, M, **synfire_layer(l)))
    return dict(
        name="cfg2", workload=f"dense LIF TTFS MLP 784-800-800-10, B={batch}, M={M}, tau=(0.5,0.25), synfire CE+T+Q",
        batch=batch, in_shape=(784,), loss="ce", tau_soft=SYNFIRE["tau_soft"], n_classes=10,
        inputs=lambda seed=SEED_INPUT, B=batch: synth.intensity_spikes(seed, (B, 784), 0.6, SYNFIRE["tau_in"]),
        labels=lambda seed=SEED_LABELS, B=batch: synth.labels(seed, B, 10),
        layers=layers)


def config3(N, M, batch=128, tau=(0.4, 0.2)):
    """One dense layer N -> N, B = 128, M steps over [0, 1], (tau_m, tau_s) = (0.4, 0.2).

    Inputs U[0, 1) with 10% silent; W = mu + N(0, 1/N) with mu N = 17.4;
    loss = sum of the output spike times that fire (one fwd+bwd pass).
    """
    W = synth.normal_weights(SEED_W + 1, (N, N), CFG3_MU_TIMES_N / N, 1.0 / math.sqrt(N))
    return dict(
        name=f"cfg3_N{N}_M{M}", workload=f"dense LIF layer {N}->{N}, B={batch}, M={M}, tau={tau}",
        batch=batch, in_shape=(N,), loss="sum_t", tau_soft=None,
        inputs=lambda seed=SEED_INPUT, B=batch: synth.uniform_spikes(seed, (B, N), 0.0, 1.0, 0.1),
        layers=[_dense(W, tau[0], tau[1], M, 0.0, 1.0)])


def _conv(W, tau_v, tau_I, M, stride, in_shape, **kw):
    d = _dense(W, tau_v, tau_I, M, **kw)
    d.update(kind="conv", stride=stride, pad=1, in_shape=tuple(in_shape))
    return d


def conv_stack(in_shape, channels, strides, n_classes, tau, M, mus, seed_w=SEED_W):
    """3x3 conv layers (pad 1, i.e. silent padding) then a dense readout.

    Layer l (1-based) has W = mu_l + N(0, 1/fan_in), fan_in = C_in * 9 for a
    conv layer and the flattened (C, H, W) size for the readout, and the
    synfire window of layer l. Returns the layer dicts and the output shape
    of every layer.
    """
    C, H, Wd = in_shape
    layers, shapes = [], []
    for l, (co, st) in enumerate(zip(channels, strides), start=1):
        W = synth.normal_weights(seed_w + l, (co, C, 3, 3), mus[l - 1], 1.0 / math.sqrt(C * 9))
        layers.append(_conv(W, tau[0], tau[1], M, st, (C, H, Wd), **synfire_layer(l)))
        H, Wd = (H + 2 - 3) // st + 1, (Wd + 2 - 3) // st + 1
        C = co
        shapes.append((C, H, Wd))
    l = len(channels) + 1
    n_in = C * H * Wd
    W = synth.normal_weights(seed_w + l, (n_classes, n_in), mus[l - 1], 1.0 / math.sqrt(n_in))
    layers.append(_dense(W, tau[0], tau[1], M, **synfire_layer(l)))
    shapes.append((n_classes,))
    return layers, shapes


def config4(batch=128, M=32):
    """9-layer conv TTFS SNN on 32x32x3 inputs (Syn-SNN-9 shapes), B = 128, M = 32.

    3x3 convs with channels 64-64-128-128-256-256-512-512, stride 2 at layers
    2, 4 and 6 (32 -> 16 -> 8 -> 4), then a dense 8192 -> 10 readout;
    (tau_m, tau_s) = (inf, inf); pixels x ~ U[0,1), t = 1 - x; bf16 operands
    with fp32 accumulation and state; CE + T + Q with AdamW.
    """
    chans = [64, 64, 128, 128, 256, 256, 512, 512]
    strides = [1, 2, 1, 2, 1, 2, 1, 1]
    layers, shapes = conv_stack((3, 32, 32), chans, strides, 10, (INF, INF), M, CFG4_MU)
    return dict(
        name="cfg4", workload=f"conv LIF TTFS SNN 9 layers on 32x32x3, B={batch}, M={M}, tau=(inf,inf), bf16",
        batch=batch, in_shape=(3, 32, 32), loss="ce", tau_soft=SYNFIRE["tau_soft"], n_classes=10, math="bf16",
        inputs=lambda seed=SEED_INPUT, B=batch: synth.intensity_spikes(seed, (B, 3, 32, 32), 0.0, SYNFIRE["tau_in"]),
        labels=lambda seed=SEED_LABELS, B=batch: synth.labels(seed, B, 10),
        layers=layers, shapes=shapes)


def config5(batch=256, M=64):
    """20-layer conv TTFS SNN on 28x28x1 inputs (Syn-SNN-20 shapes), B = 256, M = 64.

    19 3x3 convs with 64 channels (layers 1-6), 128 (7-13) and 256 (14-19),
    stride 2 at layers 7 and 14 (28 -> 14 -> 7), then a dense 12544 -> 10
    readout; (tau_m, tau_s) = (1.0, 0.25) = (4 tau_s, tau_s); staggered
    synfire windows (tau_shift = 0.1); pixels x ~ U[0,1), t = 1 - x; bf16
    operands; CE + T + Q with AdamW.
    """
    chans = [64] * 6 + [128] * 7 + [256] * 6
    strides = [1] * 6 + [2] + [1] * 6 + [2] + [1] * 5
    layers, shapes = conv_stack((1, 28, 28), chans, strides, 10, (1.0, 0.25), M, CFG5_MU)
    return dict(
        name="cfg5", workload=f"conv LIF TTFS SNN 20 layers on 28x28x1, B={batch}, M={M}, tau=(1.0,0.25), bf16",
        batch=batch, in_shape=(1, 28, 28), loss="ce", tau_soft=SYNFIRE["tau_soft"], n_classes=10, math="bf16",
        inputs=lambda seed=SEED_INPUT, B=batch: synth.intensity_spikes(seed, (B, 1, 28, 28), 0.0, SYNFIRE["tau_in"]),
        labels=lambda seed=SEED_LABELS, B=batch: synth.labels(seed, B, 10),
        layers=layers, shapes=shapes)


def _conv_k(W, tau, M, l, stride, pad, in_shape, skip=None):
    d = _conv(W, tau[0], tau[1], M, stride, in_shape, **synfire_layer(l))
    d["pad"] = pad
    if skip is not None:
        d["skip"] = skip
    return d


def syn_snn9(N=64, batch=50, M=20, tau=(INF, INF), mus=None):
    """Syn-SNN-9 of Tab. architectures on 32x32 colour images:
    C(N,3,1)-C(N,3,1)-C(N,3,1)-C(N,3,2)-C(2N,3,1)-C(2N,3,1)-C(2N,3,2)-C(2N,5,1)-10,
    with the input channels doubled (x and 1 - x, App. C.2: 6 input
    channels); zero-spike padding keeps the size ("same" padding, pad = k // 2):
    32 -> 16 (layer 4) -> 8 (layer 7), readout 2N*8*8 -> 10. Batch 50 and
    (tau_m, tau_s) = (inf, inf) as in the paper's experiments; M = 20."""
    mus = SYN9_MU if mus is None else mus
    spec = [(N, 3, 1), (N, 3, 1), (N, 3, 1), (N, 3, 2), (2 * N, 3, 1), (2 * N, 3, 1), (2 * N, 3, 2), (2 * N, 5, 1)]
    C, H = 6, 32
    layers, shapes = [], []
    for l, (co, k, st) in enumerate(spec, start=1):
        W = synth.normal_weights(SEED_W + l, (co, C, k, k), mus[l - 1], 1.0 / math.sqrt(C * k * k))
        layers.append(_conv_k(W, tau, M, l, st, k // 2, (C, H, H)))
        H = (H + 2 * (k // 2) - k) // st + 1
        C = co
        shapes.append((C, H, H))
    l = len(spec) + 1
    W = synth.normal_weights(SEED_W + l, (10, C * H * H), mus[l - 1], 1.0 / math.sqrt(C * H * H))
    layers.append(_dense(W, tau[0], tau[1], M, **synfire_layer(l)))
    shapes.append((10,))
    return dict(
        name="syn_snn9", workload=f"Syn-SNN-9 (Tab. architectures), N={N}, 32x32x6 input, B={batch}, M={M}, "
                                  f"tau=({tau[0]},{tau[1]}), bf16",
        batch=batch, in_shape=(6, 32, 32), loss="ce", tau_soft=SYNFIRE["tau_soft"], n_classes=10, math="bf16",
        inputs=lambda seed=SEED_INPUT, B=batch: synth.doubled_intensity_spikes(seed, (B, 3, 32, 32), SYNFIRE["tau_in"]),
        labels=lambda seed=SEED_LABELS, B=batch: synth.labels(seed, B, 10),
        layers=layers, shapes=shapes)


def syn_snn20(N=64, batch=50, M=20, tau=(INF, INF), mus=None, size=28, C_in=1):
    """Syn-SNN-20 of Tab. architectures on 28x28 grey images:
    C(N,3,1)-SD2(N)-SD1(N)-SD2(2N)-SD1(2N)-SD2(4N)-SD1(4N)-10.
    A skip-and-delay block (Fig. skip_connection) is three 3x3 conv layers;
    the third sees the block's input, delayed by 2 tau_shift, beside the
    second layer's output (channels concatenated, the delayed input first).
    In SD2 all three keep N channels and stride 1; in SD1 the third has
    stride 2 and 2N channels: 28 -> 14 -> 7 -> 4, readout 8N*4*4 -> 10.
    Batch 50, (tau_m, tau_s) = (inf, inf); M = 20."""
    mus = SYN20_MU if mus is None else mus
    spec = [(N, 1, None)]                       # (C_out, stride, skip source) per conv layer
    width = N
    for kind, mult in (("SD2", 1), ("SD1", 1), ("SD2", 2), ("SD1", 2), ("SD2", 4), ("SD1", 4)):
        w = N * mult
        src = len(spec) - 1                     # index of the block's input layer
        spec += [(w, 1, None), (w, 1, None), (2 * w if kind == "SD1" else w, 2 if kind == "SD1" else 1, src)]
    delay = 2 * SYNFIRE["tau_shift"]
    C, H = C_in, size
    layers, shapes, outs = [], [], []
    for l, (co, st, src) in enumerate(spec, start=1):
        cin = C + (outs[src][0] if src is not None else 0)
        W = synth.normal_weights(SEED_W + l, (co, cin, 3, 3), mus[l - 1], 1.0 / math.sqrt(cin * 9))
        layers.append(_conv_k(W, tau, M, l, st, 1, (cin, H, H), None if src is None else (src, delay)))
        H = (H + 2 - 3) // st + 1
        C = co
        outs.append((C, H, H))
        shapes.append((C, H, H))
    l = len(spec) + 1
    W = synth.normal_weights(SEED_W + l, (10, C * H * H), mus[l - 1], 1.0 / math.sqrt(C * H * H))
    layers.append(_dense(W, tau[0], tau[1], M, **synfire_layer(l)))
    shapes.append((10,))
    return dict(
        name="syn_snn20", workload=f"Syn-SNN-20 (Tab. architectures, skip-and-delay blocks), N={N}, "
                                   f"{size}x{size}x{C_in} input, B={batch}, M={M}, tau=({tau[0]},{tau[1]}), bf16",
        batch=batch, in_shape=(C_in, size, size), loss="ce", tau_soft=SYNFIRE["tau_soft"], n_classes=10, math="bf16",
        inputs=lambda seed=SEED_INPUT, B=batch: synth.intensity_spikes(seed, (B, C_in, size, size), 0.0,
                                                                       SYNFIRE["tau_in"]),
        labels=lambda seed=SEED_LABELS, B=batch: synth.labels(seed, B, 10),
        layers=layers, shapes=shapes)


def draw_offsets(layers, seed=SEED_OFFSET):
    """Per-layer t_offset draws (Alg. 2), returned as a list."""
    dts = [(L["t_end"] - L["t_first"]) / L["M"] for L in layers]
    return synth.t_offsets(seed, dts)


def with_offsets(cfg, offsets):
    """Copy of cfg whose layers carry the given t_offsets."""
    out = dict(cfg)
    out["layers"] = [dict(L, t_offset=float(o)) for L, o in zip(cfg["layers"], offsets)]
    return out


def t_max(layer):
    """Length of a layer's DSTD window (the time scale of its tolerances)."""
    return layer["t_end"] - layer["t_first"]


def as_float32_layer(layer):
    """The layer with weights rounded to float32, as the CUDA path sees them."""
    out = dict(layer)
    out["W"] = np.asarray(layer["W"], np.float32).astype(np.float64)
    return out
