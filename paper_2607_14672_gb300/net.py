"""Multi-layer driver over the C-ABI: the Alg. 2 layer loop, the loss of
Eq. cost_function and the reverse pass, with persistent device buffers.

Every step of the hot path runs in libdstd's kernels; this module only owns
the torch buffers, orders the C calls, and can capture a whole training step
in a CUDA graph (buffers never move, so a captured step replays on new data
copied into ``t_in``).
"""

import torch

from . import dstd


def narrow_layer(n_in, n_out, M, math_mode):
    """True when the library runs this dense layer on its few-output CUDA-core
    path (one kernel each way): the same test as the library's, including the
    shared memory its forward needs (W transposed, the sorted inputs)."""
    if n_out > 32 or n_in > 4096 or M > 94 or math_mode not in ("x3", "f32"):
        return False
    Mp = max(8, 1 << (M - 1).bit_length())
    nk = M + 2
    smem = 4 * (n_in * n_out + n_out * Mp + n_out) + 4 * (16 * nk + nk + 1 + 2 * n_in + 1) + 8 * n_in + 16
    return smem <= 200 * 1024


class DenseNet:
    """A stack of dense DSTD layers (configs.py layer dicts) on one GPU."""

    def __init__(self, cfg, math_mode="x3", batch=None, device="cuda", with_adamw=False):
        self.cfg = cfg
        self.math = math_mode
        self.B = int(batch or cfg["batch"])
        self.layers = [dict(L) for L in cfg["layers"]]
        self.loss_kind = cfg.get("loss", "sum_t")
        dev = torch.device(device)
        self.device = dev
        B = self.B
        self.W = [torch.tensor(L["W"], dtype=torch.float32, device=dev).contiguous() for L in self.layers]
        self.sizes = [self.W[0].shape[1]] + [w.shape[0] for w in self.W]
        self.p = [dstd.params(L, penalty_norm=1.0 / B) for L in self.layers]
        self.t_in = torch.full((B, self.sizes[0]), float("inf"), dtype=torch.float32, device=dev)
        self.t = [torch.empty((B, n), dtype=torch.float32, device=dev) for n in self.sizes[1:]]
        self.g = [torch.zeros((B, n), dtype=torch.float32, device=dev) for n in self.sizes[1:]]
        self.saved = [torch.empty(dstd.dense_saved_bytes(B, n), dtype=torch.uint8, device=dev)
                      for n in self.sizes[1:]]
        self.penalty = torch.zeros((len(self.W), 4), dtype=torch.float32, device=dev)
        self.gW = [torch.empty_like(w) for w in self.W]
        ws = max(dstd.dense_workspace_bytes(B, self.sizes[l], self.sizes[l + 1], self.p[l], math_mode)
                 for l in range(len(self.W)))
        if ws == 0:
            raise ValueError("unsupported layer sizes or constants for the library")
        self.workspace = torch.empty(ws, dtype=torch.uint8, device=dev)
        # (loss value, scratch of the fused output-layer loss: zero between calls)
        self.loss = torch.zeros(2, dtype=torch.float32, device=dev)
        self.labels = torch.zeros(B, dtype=torch.int32, device=dev)
        self.with_adamw = with_adamw
        if with_adamw:
            self.m = [torch.zeros_like(w) for w in self.W]
            self.v = [torch.zeros_like(w) for w in self.W]
            # (updates done, kernel scratch): advanced on the device by each AdamW launch
            self.adam_state = torch.zeros(2, dtype=torch.int32, device=dev)

    # -- inputs -----------------------------------------------------------
    def set_offsets(self, offsets):
        for p, L, o in zip(self.p, self.layers, offsets):
            p.t_offset = float(o)
            L["t_offset"] = float(o)

    def set_inputs(self, t0, labels=None):
        self.t_in.copy_(torch.as_tensor(t0, dtype=torch.float32), non_blocking=True)
        if labels is not None:
            self.labels.copy_(torch.as_tensor(labels, dtype=torch.int32), non_blocking=True)

    # -- passes -------------------------------------------------------------
    def layer_input(self, l):
        return self.t_in if l == 0 else self.t[l - 1]

    def forward(self, stream=None):
        for l in range(len(self.W)):
            dstd.dense_fwd(self.layer_input(l), self.W[l], self.p[l], self.math, self.t[l], self.saved[l],
                           self.penalty[l], self.workspace, stream)

    def loss_grad(self, stream=None):
        if self.loss_kind == "ce":
            dstd.ce_loss(self.t[-1], self.labels, self.cfg["tau_soft"], self.layers[-1]["t_end"], self.loss,
                         self.g[-1], stream)
        else:
            dstd.sum_t_loss(self.t[-1], self.loss, self.g[-1], stream)

    def forward_loss(self, stream=None):
        """forward, then the loss; with the CE loss the output layer and the
        loss are one library call (one kernel when the layer has few outputs)."""
        if self.loss_kind != "ce":
            self.forward(stream)
            self.loss_grad(stream)
            return
        L = len(self.W)
        for l in range(L - 1):
            dstd.dense_fwd(self.layer_input(l), self.W[l], self.p[l], self.math, self.t[l], self.saved[l],
                           self.penalty[l], self.workspace, stream)
        dstd.dense_fwd_ce(self.layer_input(L - 1), self.W[L - 1], self.p[L - 1], self.math, self.t[L - 1],
                          self.saved[L - 1], self.penalty[L - 1], self.workspace, self.labels, self.cfg["tau_soft"],
                          self.layers[-1]["t_end"], self.loss, self.g[L - 1], stream)

    def backward(self, stream=None):
        for l in range(len(self.W) - 1, -1, -1):
            g_in = self.g[l - 1] if l > 0 else None
            dstd.dense_bwd(self.layer_input(l), self.W[l], self.t[l], self.saved[l], self.g[l], self.p[l],
                           self.math, g_in, self.gW[l], self.workspace, stream)

    def optimizer(self, lr=1e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=1e-2, stream=None):
        dstd.adamw_multi(self.W, self.gW, self.m, self.v, lr, betas[0], betas[1], eps, weight_decay,
                         self.adam_state, None, stream)

    def step(self, stream=None):
        """One training step: forward, loss, backward (and AdamW if enabled)."""
        self.forward_loss(stream)
        self.backward(stream)
        if self.with_adamw:
            self.optimizer(stream=stream)

    def objective(self):
        """Eq. cost_function on the last batch: loss + T + gamma_Q Q (device scalar)."""
        return self.loss[0] + self.penalty[:, 0].sum() + self.penalty[:, 1].sum()

    def launches_per_step(self):
        """Kernels the library launches per ``step`` (memsets not counted)."""
        tc = self.math != "f32"
        L = len(self.W)
        fused_loss = self.loss_kind == "ce" and narrow_layer(self.sizes[-2], self.sizes[-1], self.layers[-1]["M"],
                                                             self.math)
        n = 0 if fused_loss else 1                # loss (inside the output layer's kernel when fused)
        for l in range(L):
            n_in, n_out = self.sizes[l], self.sizes[l + 1]
            if narrow_layer(n_in, n_out, self.layers[l]["M"], self.math):
                n += 2                            # few outputs: one fused kernel each way (CUDA cores)
                continue
            n += 3 if self.math == "x3" else 4    # fwd: [prep +] binning (x3: one launch for both) + gemm + scan
            n += 3 if tc else 4                   # bwd: dw^ + binning^T + dW gemm [+ split-K reduce]
            if l > 0:                             # bwd input times: prep W^T + dS gemm [+ gather]
                n += 2 if tc else 3
        if self.with_adamw:
            n += 1                                # one AdamW launch for all layers
        return n


class ConvNet:
    """A stack of conv DSTD layers and a dense readout (configs 4 and 5) on one GPU.

    Spike tensors are NHWC ([B, H, W, C]); filters are kept as [C_out, k, k,
    C_in]. The layer dicts hold oracle-layout weights ([C_out, C_in, k, k]
    filters; the readout's columns in (C, H, W) order), which the constructor
    permutes once, so both sides compute the same network. T and Q of a conv
    layer are normalised by B Ho Wo (App. C.1).
    """

    def __init__(self, cfg, math_mode=None, batch=None, device="cuda", with_adamw=True):
        self.cfg = cfg
        self.math = math_mode or cfg.get("math", "bf16")
        self.B = B = int(batch or cfg["batch"])
        self.layers = [dict(L) for L in cfg["layers"]]
        dev = torch.device(device)
        self.device = dev
        C, H, Wd = cfg["in_shape"]
        self.in_shape = (H, Wd, C)
        self.W, self.p, self.t, self.g, self.saved, self.geom = [], [], [], [], [], []
        # skip-and-delay layers (App. C.3): per layer, (source layer or -1, delay,
        # concatenated input, its gradient), else None
        self.skip = []
        ws = 0
        shape = (H, Wd, C)
        for l, L in enumerate(self.layers):
            Wl = torch.tensor(L["W"], dtype=torch.float32)
            sk = L.get("skip")
            if sk is not None:
                src, delay = int(sk[0]), float(sk[1])
                s_shape = (H, Wd, C) if src < 0 else tuple(self.t[src].shape[1:])
                if s_shape[:2] != shape[:2]:
                    raise ValueError(f"layer {l}: skip source and previous output differ in size")
                shape = (shape[0], shape[1], s_shape[2] + shape[2])
                cat = torch.empty((B,) + shape, dtype=torch.float32, device=dev)
                self.skip.append((src, delay, cat, torch.empty_like(cat), s_shape[2]))
            else:
                self.skip.append(None)
            if L["kind"] == "conv":
                Hh, Ww, Cc = shape
                k, st, pad = Wl.shape[2], L["stride"], L["pad"]
                Ho, Wo = dstd.conv_out_hw(Hh, Ww, k, st, pad)
                Co = Wl.shape[0]
                self.W.append(Wl.permute(0, 2, 3, 1).contiguous().to(dev))
                p = dstd.params(L, penalty_norm=1.0 / (B * Ho * Wo))
                need = dstd.conv_workspace_bytes(B, Hh, Ww, Cc, Co, k, st, pad, p, self.math)
                self.geom.append((Hh, Ww, Cc, k, st, pad))
                shape = (Ho, Wo, Co)
                self.saved.append(torch.empty(dstd.dense_saved_bytes(B * Ho * Wo, Co), dtype=torch.uint8, device=dev))
            else:
                Hh, Ww, Cc = shape
                n_out = Wl.shape[0]
                # readout columns: oracle order (c, y, x) -> NHWC order (y, x, c)
                Wl = Wl.reshape(n_out, Cc, Hh, Ww).permute(0, 2, 3, 1).reshape(n_out, -1) if Hh * Ww > 1 else Wl
                self.W.append(Wl.contiguous().to(dev))
                p = dstd.params(L, penalty_norm=1.0 / B)
                need = dstd.dense_workspace_bytes(B, Hh * Ww * Cc, n_out, p, self.math)
                self.geom.append(None)
                shape = (n_out,)
                self.saved.append(torch.empty(dstd.dense_saved_bytes(B, n_out), dtype=torch.uint8, device=dev))
            if need == 0:
                raise ValueError("unsupported layer sizes or constants for the library")
            ws = max(ws, need)
            self.p.append(p)
            self.t.append(torch.empty((B,) + shape, dtype=torch.float32, device=dev))
            self.g.append(torch.zeros((B,) + shape, dtype=torch.float32, device=dev))
        self.t_in = torch.full((B, H, Wd, C), float("inf"), dtype=torch.float32, device=dev)
        self.penalty = torch.zeros((len(self.W), 4), dtype=torch.float32, device=dev)
        self.gW = [torch.empty_like(w) for w in self.W]
        self.workspace = torch.empty(ws, dtype=torch.uint8, device=dev)
        self.loss = torch.zeros(1, dtype=torch.float32, device=dev)
        self.labels = torch.zeros(B, dtype=torch.int32, device=dev)
        self.with_adamw = with_adamw
        if with_adamw:
            self.m = [torch.zeros_like(w) for w in self.W]
            self.v = [torch.zeros_like(w) for w in self.W]
            # (updates done, kernel scratch): advanced on the device by each AdamW launch
            self.adam_state = torch.zeros(2, dtype=torch.int32, device=dev)

    def set_offsets(self, offsets):
        for p, L, o in zip(self.p, self.layers, offsets):
            p.t_offset = float(o)
            L["t_offset"] = float(o)

    def set_inputs(self, t0, labels=None):
        """t0 in the oracle's [B, C, H, W] layout (or already NHWC via ``set_inputs_nhwc``)."""
        x = torch.as_tensor(t0, dtype=torch.float32)
        self.t_in.copy_(x.permute(0, 2, 3, 1), non_blocking=True)
        if labels is not None:
            self.labels.copy_(torch.as_tensor(labels, dtype=torch.int32), non_blocking=True)

    def layer_input(self, l):
        if self.skip[l] is not None:
            return self.skip[l][2]
        return self.t_in if l == 0 else self.t[l - 1]

    def forward(self, stream=None):
        for l, L in enumerate(self.layers):
            sk = self.skip[l]
            if sk is not None:
                src, delay, cat = sk[0], sk[1], sk[2]
                dstd.concat_channels(self.t_in if src < 0 else self.t[src], self.t_in if l == 0 else self.t[l - 1],
                                     delay, cat, stream)
            x = self.layer_input(l)
            if self.geom[l] is not None:
                _, _, _, k, st, pad = self.geom[l]
                dstd.conv_fwd(x, self.W[l], st, pad, self.p[l], self.math, self.t[l], self.saved[l],
                              self.penalty[l], self.workspace, stream)
            else:
                dstd.dense_fwd(x.reshape(self.B, -1), self.W[l], self.p[l], self.math, self.t[l], self.saved[l],
                               self.penalty[l], self.workspace, stream)

    def loss_grad(self, stream=None):
        dstd.ce_loss(self.t[-1], self.labels, self.cfg["tau_soft"], self.layers[-1]["t_end"], self.loss,
                     self.g[-1], stream)

    def backward(self, stream=None):
        """Layers in reverse. A layer's input gradient overwrites the previous
        output's; a skip layer's goes to its concatenated input and is split:
        the previous layer's part overwrites, and the delayed source's part
        is added into the source's gradient once the layer after the source
        (the block's first layer) has written it."""
        for l in range(len(self.layers) - 1, -1, -1):
            x = self.layer_input(l)
            sk = self.skip[l]
            if sk is not None:
                g_in = sk[3]
            else:
                g_in = self.g[l - 1] if l > 0 else None
            if self.geom[l] is not None:
                _, _, _, k, st, pad = self.geom[l]
                dstd.conv_bwd(x, self.W[l], self.t[l], self.saved[l], self.g[l], st, pad, self.p[l], self.math,
                              g_in, self.gW[l], self.workspace, stream)
            else:
                dstd.dense_bwd(x.reshape(self.B, -1), self.W[l], self.t[l], self.saved[l], self.g[l], self.p[l],
                               self.math, None if g_in is None else g_in.reshape(self.B, -1), self.gW[l],
                               self.workspace, stream)
            if sk is not None and l > 0:
                dstd.split_channels(sk[3], sk[4], g_b=self.g[l - 1], stream=stream)
            # skip layers that read the output of layer l - 1: add their part now
            for m in range(l, len(self.layers)):
                sm = self.skip[m]
                if sm is not None and sm[0] == l - 1 and l > 0:
                    dstd.split_channels(sm[3], sm[4], g_a=self.g[l - 1], accumulate_a=True, stream=stream)

    def optimizer(self, lr=1e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=1e-2, stream=None):
        dstd.adamw_multi(self.W, self.gW, self.m, self.v, lr, betas[0], betas[1], eps, weight_decay,
                         self.adam_state, None, stream)

    def step(self, stream=None):
        """One training step: forward, loss, backward, AdamW."""
        self.forward(stream)
        self.loss_grad(stream)
        self.backward(stream)
        if self.with_adamw:
            self.optimizer(stream=stream)

    def objective(self):
        return self.loss[0] + self.penalty[:, 0].sum() + self.penalty[:, 1].sum()

    def dead_fraction(self):
        """Share of silent neurons per layer on the last batch (from the Q counters)."""
        pen = self.penalty.detach().cpu()
        return (pen[:, 2] / (pen[:, 2] + pen[:, 3]).clamp(min=1.0)).tolist()
