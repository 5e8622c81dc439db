"""Oracle, training objective and optimizer (App. C.1).

Test infrastructure (see the package header). Float64 throughout.

Parity status: pinned. Every gradient against central finite differences of
its value; AdamW against ``torch.optim.AdamW`` (a library routine with the
same definition); the warm-up schedule against its closed form
eta(p) = eta_0 2^{min(p, N_warm) - N_warm}.

Cost (Eq. cost_function), per sample and averaged over the mini-batch:
    C = L(t^(L) | kappa) + T({t^(l)}) + gamma_Q Q
  L  cross-entropy of the target over S_i = softmax(-t_i^(L) / tau_soft).
  T  temporal penalty (Eq. temporal_penalty): per layer l and neuron i,
       gamma_head (t - t_head^(l))^2 theta(t_head^(l) - t)
     + gamma_tail (t - t_tail^(l))^2 theta(t - t_tail^(l)),
     t_head^(l) = l tau_shift + t_head, t_tail^(l) = l tau_shift + tau_width - t_tail.
  Q  dead-neuron term (Eq. dead_neuron_penalty): -sum_{i,l} 1{t_i = inf} sum_j w_ij.
  For convolutional layers T and Q are divided by the spatial size.

Readings where the paper is silent (the CUDA path takes the same ones):
  R7  T skips silent neurons (the paper notes T gives them no gradient);
      in L a silent output enters with the constant time ``t_silent`` (the
      output layer's window end), so the loss stays finite and a silent
      output passes no gradient.
"""

import numpy as np

INF = np.inf


def window_params(l, tau_shift, tau_width, tau_margin, t_head, t_tail):
    """Per-layer synfire constants (App. C.1), layer index l >= 1.

    Returns dict with t_head_l, t_tail_l (Eq. temporal_penalty) and the DSTD
    window t_first = l tau_shift - tau_margin, t_end = l tau_shift +
    tau_width + tau_margin.
    """
    return {
        "t_head_l": l * tau_shift + t_head,
        "t_tail_l": l * tau_shift + tau_width - t_tail,
        "t_first": l * tau_shift - tau_margin,
        "t_end": l * tau_shift + tau_width + tau_margin,
    }


def ce_loss(t_L, labels, tau_soft, t_silent):
    """Mini-batch mean cross-entropy over softmax(-t / tau_soft).

    t_L [B, C] output spike times, labels [B] integer targets (one-hot kappa).
    Returns (loss, g_t_L [B, C]) with g = d loss / d t_L.
    """
    t_L = np.asarray(t_L, float)
    B = t_L.shape[0]
    silent = ~np.isfinite(t_L)
    t_eff = np.where(silent, t_silent, t_L)
    z = -t_eff / tau_soft
    z = z - z.max(-1, keepdims=True)
    p = np.exp(z)
    p = p / p.sum(-1, keepdims=True)
    idx = np.arange(B)
    loss = -np.mean(np.log(p[idx, labels]))
    kap = np.zeros_like(p)
    kap[idx, labels] = 1.0
    # dL/dz = S - kappa, dz/dt = -1/tau_soft; batch mean
    g = -(p - kap) / tau_soft / B
    return loss, np.where(silent, 0.0, g)


def temporal_penalty(t, t_head_l, t_tail_l, gamma_head, gamma_tail, norm):
    """T of one layer times ``norm`` (1/B, or 1/(B H W) for conv layers).

    t [B, ...] spike times. Returns (value, d value / d t).
    """
    t = np.asarray(t, float)
    fired = np.isfinite(t)
    tf = np.where(fired, t, 0.0)
    head = (tf < t_head_l) & fired
    tail = (tf > t_tail_l) & fired
    val = np.sum(np.where(head, gamma_head * (tf - t_head_l) ** 2, 0.0)
                 + np.where(tail, gamma_tail * (tf - t_tail_l) ** 2, 0.0))
    g = np.where(head, 2 * gamma_head * (tf - t_head_l), 0.0) + \
        np.where(tail, 2 * gamma_tail * (tf - t_tail_l), 0.0)
    return norm * val, norm * g


def dead_neuron_penalty(t, W_rowsum, gamma_q, norm):
    """gamma_Q Q of one layer times ``norm``, and its gradient w.r.t. W.

    t [B, N] spike times of the layer's neurons, W_rowsum [N] = sum_j w_ij
    (for conv: the sum over the whole filter of the neuron's channel).
    Returns (value, count [N]) where d value / d w_ij = -gamma_q norm count_i.
    """
    silent = ~np.isfinite(np.asarray(t, float))
    count = silent.sum(0).astype(float)
    val = -gamma_q * norm * np.sum(count * np.asarray(W_rowsum, float))
    return val, count


def adamw_step(w, g, m, v, step, lr, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=1e-2):
    """One AdamW update (decoupled weight decay, Loshchilov & Hutter).

    step is the 1-based update count. Returns new (w, m, v).
    """
    w = np.asarray(w, float) * (1.0 - lr * weight_decay)
    m = beta1 * np.asarray(m, float) + (1 - beta1) * g
    v = beta2 * np.asarray(v, float) + (1 - beta2) * g * g
    mh = m / (1 - beta1 ** step)
    vh = v / (1 - beta2 ** step)
    return w - lr * mh / (np.sqrt(vh) + eps), m, v


def warmup_lr(p, eta0, n_warm):
    """Learning rate at epoch p: eta(0) = eta_0 / 2^N_warm, doubling each
    epoch while p < N_warm, constant afterwards (App. C.1)."""
    eta = eta0 / 2.0 ** n_warm
    for q in range(p):
        if q < n_warm:
            eta *= 2.0
    return eta
