"""Thin Python binding of libdstd (include/dstd.h): argument marshalling only.

Every function takes CUDA float32 torch tensors (int32 for labels, any dtype
for opaque byte buffers), checks shapes and dtypes, and calls the C entry
point of the same name on the given stream (default: torch's current
stream). All arithmetic happens in the library's kernels; there is no
fallback of any kind. A missing library raises at load time.
"""

import ctypes
import os

from .build import LIB_PATH

MATH = {"f32": 0, "x3": 1, "bf16": 2}

ERRORS = {0: "ok", -1: "invalid argument", -2: "unsupported size or mode", -3: "workspace too small",
          -4: "CUDA call or kernel launch failed", -5: "a bounded device-side wait expired",
          -6: "no usable sm_103 device"}

EXPORTS = ("dstd_dense_saved_bytes", "dstd_dense_workspace_bytes", "dstd_binning", "dstd_dense_what",
           "dstd_scan_solve", "dstd_dense_fwd", "dstd_dense_fwd_ce", "dstd_dense_bwd", "dstd_ce_loss", "dstd_sum_t_loss",
           "dstd_adamw", "dstd_adamw_multi", "dstd_device_status", "dstd_error_string", "dstd_version", "dstd_timing_enable",
           "dstd_timing_read", "dstd_timing_collect", "dstd_set_pair_policy", "dstd_conv_set_chunk_images", "dstd_conv_set_operand_policy", "dstd_kernel_kind_count", "dstd_kernel_kind_name", "dstd_selftest_wait_timeout",
           "dstd_dense_fwd_noalloc", "dstd_conv_workspace_bytes", "dstd_conv_fwd", "dstd_conv_bwd",
           "dstd_exact_workspace_bytes", "dstd_exact_fwd", "dstd_exact_bwd", "dstd_concat_channels", "dstd_split_channels",
           "dstd_ms_saved_bytes", "dstd_ms_workspace_bytes", "dstd_dense_fwd_ms", "dstd_dense_bwd_ms")


class DstdError(RuntimeError):
    def __init__(self, code, where):
        super().__init__(f"{where}: {ERRORS.get(code, 'unknown error')} (code {code})")
        self.code = code


class Params(ctypes.Structure):
    """dstd_params of include/dstd.h."""
    _fields_ = [("tau_m", ctypes.c_float), ("tau_s", ctypes.c_float), ("v_th", ctypes.c_float),
                ("t_first", ctypes.c_float), ("t_end", ctypes.c_float), ("M", ctypes.c_int32),
                ("t_offset", ctypes.c_float), ("t_head", ctypes.c_float), ("t_tail", ctypes.c_float),
                ("gamma_head", ctypes.c_float), ("gamma_tail", ctypes.c_float), ("gamma_q", ctypes.c_float),
                ("penalty_norm", ctypes.c_float)]


def params(layer, penalty_norm=0.0):
    """dstd_params from a layer dict (see configs.py)."""
    return Params(float(layer["tau_v"]), float(layer["tau_I"]), float(layer["v_th"]), float(layer["t_first"]),
                  float(layer["t_end"]), int(layer["M"]), float(layer.get("t_offset", 0.0)),
                  float(layer.get("t_head_l", 0.0)), float(layer.get("t_tail_l", 0.0)),
                  float(layer.get("gamma_head", 0.0)), float(layer.get("gamma_tail", 0.0)),
                  float(layer.get("gamma_q", 0.0)), float(penalty_norm))


_LIB = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_SZ = ctypes.c_size_t
_I64 = ctypes.c_int64
_PP = ctypes.POINTER(Params)


def load(path=None):
    """Load libdstd.so (built by ``build.build()``); raises if it is missing."""
    global _LIB
    if _LIB is not None:
        return _LIB
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"libdstd.so not found at {p}: build it first (python -m paper_2607_14672_gb300.build)")
    lib = ctypes.CDLL(p)
    sig = {
        "dstd_dense_saved_bytes": (_SZ, [_I, _I]),
        "dstd_dense_workspace_bytes": (_SZ, [_I, _I, _I, _PP, _I]),
        "dstd_binning": (_I, [_P, _I, _I, _PP, _P, _P, _P]),
        "dstd_dense_what": (_I, [_P, _P, _I, _I, _I, _PP, _I, _P, _P, _SZ, _P]),
        "dstd_scan_solve": (_I, [_P, _I, _I, _PP, _P, _P, _P, _P, _P]),
        "dstd_dense_fwd": (_I, [_P, _P, _I, _I, _I, _PP, _I, _P, _P, _P, _P, _SZ, _P]),
        "dstd_dense_fwd_ce": (_I, [_P, _P, _I, _I, _I, _PP, _I, _P, _P, _P, _P, _SZ, _P, _F, _F, _P, _P, _P]),
        "dstd_dense_bwd": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _PP, _I, _P, _P, _P, _SZ, _P]),
        "dstd_ce_loss": (_I, [_P, _P, _I, _I, _F, _F, _P, _P, _P]),
        "dstd_sum_t_loss": (_I, [_P, _I64, _P, _P, _P]),
        "dstd_adamw": (_I, [_P, _P, _P, _P, _I64, _F, _F, _F, _F, _F, _I, _P]),
        "dstd_adamw_multi": (_I, [_I, _P, _P, _P, _P, _P, _F, _F, _F, _F, _F, _P, _P, _P]),
        "dstd_device_status": (_I, [_I]),
        "dstd_error_string": (ctypes.c_char_p, [_I]),
        "dstd_version": (_I, []),
        "dstd_timing_enable": (_I, [_I]),
        "dstd_timing_read": (_I, [_I, ctypes.POINTER(_F), ctypes.POINTER(_I64)]),
        "dstd_timing_collect": (_I, []),
        "dstd_set_pair_policy": (_I, [_I]),
        "dstd_conv_set_chunk_images": (_I, [_I]),
        "dstd_conv_set_operand_policy": (_I, [_I]),
        "dstd_exact_workspace_bytes": (_SZ, [_I, _I, _I]),
        "dstd_exact_fwd": (_I, [_P, _P, _I, _I, _I, _PP, _P, _P, _SZ, _P]),
        "dstd_exact_bwd": (_I, [_P, _P, _P, _P, _I, _I, _I, _PP, _P, _P, _P, _SZ, _P]),
        "dstd_kernel_kind_count": (_I, []),
        "dstd_kernel_kind_name": (ctypes.c_char_p, [_I]),
        "dstd_selftest_wait_timeout": (_I, [ctypes.c_uint32, _P]),
        "dstd_dense_fwd_noalloc": (_I, [_P, _P, _I, _I, _I, _PP, _I, _P, _P, _P, _P]),
        "dstd_conv_workspace_bytes": (_SZ, [_I, _I, _I, _I, _I, _I, _I, _I, _PP, _I]),
        "dstd_conv_fwd": (_I, [_P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _PP, _I, _P, _P, _P, _P, _SZ, _P]),
        "dstd_conv_bwd": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _I, _PP, _I, _P, _P, _P, _SZ, _P]),
        "dstd_concat_channels": (_I, [_P, _I, _F, _P, _I, _I64, _P, _P]),
        "dstd_ms_saved_bytes": (_SZ, [_I, _I, _I]),
        "dstd_ms_workspace_bytes": (_SZ, [_I, _I, _I, _I, _I, _PP, _I]),
        "dstd_dense_fwd_ms": (_I, [_P, _P, _I, _I, _I, _I, _I, _PP, _I, _P, _P, _P, _SZ, _P]),
        "dstd_dense_bwd_ms": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _PP, _I, _P, _P, _P, _SZ, _P]),
        "dstd_split_channels": (_I, [_P, _I, _I, _I64, _P, _I, _P, _I, _P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _LIB = lib
    return lib


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _stream(stream):
    if stream is not None:
        return stream if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


def _check(code, where):
    if code != 0:
        raise DstdError(code, where)


def _f32(x, name, shape=None):
    import torch
    if x.dtype != torch.float32 or not x.is_cuda or not x.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA float32 tensor")
    if shape is not None and tuple(x.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(x.shape)}, expected {tuple(shape)}")


def version():
    return load().dstd_version()


def error_string(code):
    return load().dstd_error_string(code).decode()


def dense_saved_bytes(B, N_out):
    return load().dstd_dense_saved_bytes(B, N_out)


def dense_workspace_bytes(B, N_in, N_out, p, math_mode):
    return load().dstd_dense_workspace_bytes(B, N_in, N_out, ctypes.byref(p), MATH[math_mode])


def binning(t_in, p, s, ds=None, stream=None):
    B, N = t_in.shape
    _f32(t_in, "t_in")
    _f32(s, "s", (B, p.M, N))
    if ds is not None:
        _f32(ds, "ds", (B, p.M, N))
    _check(load().dstd_binning(_ptr(t_in), B, N, ctypes.byref(p), _ptr(s), _ptr(ds), _stream(stream)),
           "dstd_binning")


def dense_what(t_in, W, p, math_mode, what, workspace, stream=None):
    B, N_in = t_in.shape
    N_out = W.shape[0]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(what, "what", (B, N_out, p.M))
    _check(load().dstd_dense_what(_ptr(t_in), _ptr(W), B, N_in, N_out, ctypes.byref(p), MATH[math_mode],
                                  _ptr(what), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                  _stream(stream)), "dstd_dense_what")


def scan_solve(what, p, w_rowsum, t_out, saved=None, penalty=None, stream=None):
    B, N_out, M = what.shape
    _f32(what, "what")
    _f32(t_out, "t_out", (B, N_out))
    _check(load().dstd_scan_solve(_ptr(what), B, N_out, ctypes.byref(p), _ptr(w_rowsum), _ptr(t_out), _ptr(saved),
                                  _ptr(penalty), _stream(stream)), "dstd_scan_solve")


def dense_fwd(t_in, W, p, math_mode, t_out, saved, penalty, workspace, stream=None):
    B, N_in = t_in.shape
    N_out = W.shape[0]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(t_out, "t_out", (B, N_out))
    _check(load().dstd_dense_fwd(_ptr(t_in), _ptr(W), B, N_in, N_out, ctypes.byref(p), MATH[math_mode], _ptr(t_out),
                                 _ptr(saved), _ptr(penalty), _ptr(workspace),
                                 workspace.numel() * workspace.element_size(), _stream(stream)), "dstd_dense_fwd")


def dense_fwd_ce(t_in, W, p, math_mode, t_out, saved, penalty, workspace, labels, tau_soft, t_silent, loss,
                 g_t_out, stream=None):
    """dense_fwd of the output layer, then the CE loss of its spike times
    (fused into one kernel on the few-output path). loss: float32[2] device
    tensor, loss[1] zero before the first call (left zero)."""
    B, N_in = t_in.shape
    N_out = W.shape[0]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(t_out, "t_out", (B, N_out))
    _f32(g_t_out, "g_t_out", (B, N_out))
    if loss.numel() < 2:
        raise ValueError("dense_fwd_ce: loss must hold 2 floats (value, scratch)")
    _check(load().dstd_dense_fwd_ce(_ptr(t_in), _ptr(W), B, N_in, N_out, ctypes.byref(p), MATH[math_mode],
                                    _ptr(t_out), _ptr(saved), _ptr(penalty), _ptr(workspace),
                                    workspace.numel() * workspace.element_size(), _ptr(labels), float(tau_soft),
                                    float(t_silent), _ptr(loss), _ptr(g_t_out), _stream(stream)), "dstd_dense_fwd_ce")


def dense_fwd_noalloc(t_in, W, p, math_mode, t_out, saved, penalty=None, stream=None):
    """dstd_dense_fwd without a workspace: for callers that cannot allocate
    device memory; scratch is the library's fixed 64 MiB device array, shared
    by every call (do not overlap calls on the GPU)."""
    B, N_in = t_in.shape
    N_out = W.shape[0]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(t_out, "t_out", (B, N_out))
    _check(load().dstd_dense_fwd_noalloc(_ptr(t_in), _ptr(W), B, N_in, N_out, ctypes.byref(p), MATH[math_mode],
                                         _ptr(t_out), _ptr(saved), _ptr(penalty), _stream(stream)),
           "dstd_dense_fwd_noalloc")


def dense_bwd(t_in, W, t_out, saved, g_t_out, p, math_mode, g_t_in, g_W, workspace, stream=None):
    B, N_in = t_in.shape
    N_out = W.shape[0]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(g_W, "g_W", (N_out, N_in))
    if g_t_in is not None:
        _f32(g_t_in, "g_t_in", (B, N_in))
    _check(load().dstd_dense_bwd(_ptr(t_in), _ptr(W), _ptr(t_out), _ptr(saved), _ptr(g_t_out), B, N_in, N_out,
                                 ctypes.byref(p), MATH[math_mode], _ptr(g_t_in), _ptr(g_W), _ptr(workspace),
                                 workspace.numel() * workspace.element_size(), _stream(stream)), "dstd_dense_bwd")


def conv_out_hw(H, W, k, stride, pad):
    return (H + 2 * pad - k) // stride + 1, (W + 2 * pad - k) // stride + 1


def conv_workspace_bytes(B, H, W, C_in, C_out, k, stride, pad, p, math_mode):
    return load().dstd_conv_workspace_bytes(B, H, W, C_in, C_out, k, stride, pad, ctypes.byref(p), MATH[math_mode])


def conv_fwd(t_in, W, stride, pad, p, math_mode, t_out, saved, penalty, workspace, stream=None):
    """t_in [B, H, W, C_in] NHWC, W [C_out, k, k, C_in] -> t_out [B, Ho, Wo, C_out]."""
    B, H, Wd, C = t_in.shape
    C_out, k = W.shape[0], W.shape[1]
    Ho, Wo = conv_out_hw(H, Wd, k, stride, pad)
    _f32(t_in, "t_in")
    _f32(W, "W", (C_out, k, k, C))
    _f32(t_out, "t_out", (B, Ho, Wo, C_out))
    _check(load().dstd_conv_fwd(_ptr(t_in), _ptr(W), B, H, Wd, C, C_out, k, stride, pad, ctypes.byref(p),
                                MATH[math_mode], _ptr(t_out), _ptr(saved), _ptr(penalty), _ptr(workspace),
                                workspace.numel() * workspace.element_size(), _stream(stream)), "dstd_conv_fwd")


def conv_bwd(t_in, W, t_out, saved, g_t_out, stride, pad, p, math_mode, g_t_in, g_W, workspace, stream=None):
    B, H, Wd, C = t_in.shape
    C_out, k = W.shape[0], W.shape[1]
    _f32(t_in, "t_in")
    _f32(W, "W", (C_out, k, k, C))
    _f32(g_W, "g_W", (C_out, k, k, C))
    if g_t_in is not None:
        _f32(g_t_in, "g_t_in", (B, H, Wd, C))
    _check(load().dstd_conv_bwd(_ptr(t_in), _ptr(W), _ptr(t_out), _ptr(saved), _ptr(g_t_out), B, H, Wd, C, C_out, k,
                                stride, pad, ctypes.byref(p), MATH[math_mode], _ptr(g_t_in), _ptr(g_W),
                                _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)),
           "dstd_conv_bwd")


def ce_loss(t_L, labels, tau_soft, t_silent, loss, g_t_L, stream=None):
    B, C = t_L.shape
    _f32(t_L, "t_L")
    _check(load().dstd_ce_loss(_ptr(t_L), _ptr(labels), B, C, float(tau_soft), float(t_silent), _ptr(loss),
                               _ptr(g_t_L), _stream(stream)), "dstd_ce_loss")


def ms_saved_bytes(B, N_out, F_out):
    return load().dstd_ms_saved_bytes(B, N_out, F_out)


def ms_workspace_bytes(B, N_in, N_out, F_in, F_out, p, math="x3"):
    return load().dstd_ms_workspace_bytes(B, N_in, N_out, F_in, F_out, ctypes.byref(p), MATH[math])


def dense_fwd_ms(t_in, W, p, math, t_out, saved, workspace, stream=None):
    """Multi-spike layer forward: t_in [B, N_in, F_in] -> t_out [B, N_out, F_out]."""
    B, N_in, F_in = t_in.shape
    N_out, F_out = t_out.shape[1], t_out.shape[2]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(t_out, "t_out", (B, N_out, F_out))
    _check(load().dstd_dense_fwd_ms(_ptr(t_in), _ptr(W), B, N_in, N_out, F_in, F_out, ctypes.byref(p), MATH[math],
                                    _ptr(t_out), _ptr(saved), _ptr(workspace), workspace.numel(), _stream(stream)),
           "dstd_dense_fwd_ms")


def dense_bwd_ms(t_in, W, t_out, saved, g_t_out, p, math, g_t_in, g_W, workspace, stream=None):
    """Multi-spike layer backward (g_t_in may be None)."""
    B, N_in, F_in = t_in.shape
    N_out, F_out = t_out.shape[1], t_out.shape[2]
    _check(load().dstd_dense_bwd_ms(_ptr(t_in), _ptr(W), _ptr(t_out), _ptr(saved), _ptr(g_t_out), B, N_in, N_out,
                                    F_in, F_out, ctypes.byref(p), MATH[math], _ptr(g_t_in), _ptr(g_W),
                                    _ptr(workspace), workspace.numel(), _stream(stream)), "dstd_dense_bwd_ms")


def concat_channels(a, b, delay_a, out, stream=None):
    """out[..., :C_a] = a + delay_a, out[..., C_a:] = b (channels innermost)."""
    for x, nm in ((a, "a"), (b, "b"), (out, "out")):
        _f32(x, nm)
    Ca, Cb = a.shape[-1], b.shape[-1]
    P = a.numel() // Ca
    if b.numel() != P * Cb or out.numel() != P * (Ca + Cb):
        raise ValueError("concat_channels: a, b and out disagree on the number of positions")
    _check(load().dstd_concat_channels(_ptr(a), Ca, float(delay_a), _ptr(b), Cb, P, _ptr(out),
                                       _stream(stream)), "dstd_concat_channels")


def split_channels(g, C_a, g_a=None, accumulate_a=False, g_b=None, accumulate_b=False, stream=None):
    """Adjoint of concat_channels: g[..., :C_a] into g_a, g[..., C_a:] into g_b
    (overwriting, or adding with accumulate_*); either target may be None."""
    _f32(g, "g")
    Ct = g.shape[-1]
    Cb = Ct - C_a
    P = g.numel() // Ct
    _check(load().dstd_split_channels(_ptr(g), int(C_a), int(Cb), P, _ptr(g_a) if g_a is not None else None,
                                      int(bool(accumulate_a)), _ptr(g_b) if g_b is not None else None,
                                      int(bool(accumulate_b)), _stream(stream)), "dstd_split_channels")


def sum_t_loss(t, loss, g, stream=None):
    _f32(t, "t")
    _check(load().dstd_sum_t_loss(_ptr(t), t.numel(), _ptr(loss), _ptr(g), _stream(stream)), "dstd_sum_t_loss")


def adamw(w, g, m, v, lr, beta1, beta2, eps, weight_decay, step, stream=None):
    _f32(w, "w")
    _check(load().dstd_adamw(_ptr(w), _ptr(g), _ptr(m), _ptr(v), w.numel(), float(lr), float(beta1), float(beta2),
                             float(eps), float(weight_decay), int(step), _stream(stream)), "dstd_adamw")


def adamw_multi(ws, gs, ms, vs, lr, beta1, beta2, eps, weight_decay, step, lr_dev=None, stream=None):
    """One AdamW launch over the tensors ws (in place, with gs, ms, vs alike);
    step is a device int32[2] tensor holding (updates done, 0)."""
    k = len(ws)
    if not (len(gs) == len(ms) == len(vs) == k):
        raise ValueError("adamw_multi: tensor lists differ in length")
    for w in ws:
        _f32(w, "w")
    import torch
    if step.dtype != torch.int32 or step.numel() != 2 or not step.is_cuda:
        raise ValueError("adamw_multi: step must be a device int32 tensor of 2 elements")
    arr = lambda xs: (ctypes.c_void_p * k)(*[x.data_ptr() for x in xs])
    n = (ctypes.c_int64 * k)(*[w.numel() for w in ws])
    _check(load().dstd_adamw_multi(k, arr(ws), arr(gs), arr(ms), arr(vs), n, float(lr), float(beta1), float(beta2),
                                   float(eps), float(weight_decay), _ptr(step), _ptr(lr_dev), _stream(stream)),
           "dstd_adamw_multi")


def device_status(clear=True):
    """DSTD_OK (0) or DSTD_E_TIMEOUT after synchronising the device."""
    return load().dstd_device_status(1 if clear else 0)



def timing_enable(on=True):
    """Turn per-kernel event timing on/off (clears the counters)."""
    _check(load().dstd_timing_enable(1 if on else 0), "dstd_timing_enable")


def exact_workspace_bytes(B, N_in, N_out):
    return load().dstd_exact_workspace_bytes(B, N_in, N_out)


def exact_fwd(t_in, W, p, t_out, workspace, stream=None):
    """Exact (event-driven, Alg. 1) first-spike times of a dense layer."""
    B, N_in = t_in.shape
    N_out = W.shape[0]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(t_out, "t_out", (B, N_out))
    _check(load().dstd_exact_fwd(_ptr(t_in), _ptr(W), B, N_in, N_out, ctypes.byref(p), _ptr(t_out), _ptr(workspace),
                                 workspace.numel() * workspace.element_size(), _stream(stream)), "dstd_exact_fwd")


def exact_bwd(t_in, W, t_out, g_t_out, p, g_t_in, g_W, workspace, stream=None):
    """Backward of the exact layer (implicit function theorem at each exact
    spike time): g_W [N_out, N_in] and g_t_in [B, N_in] (or None), overwritten."""
    B, N_in = t_in.shape
    N_out = W.shape[0]
    _f32(t_in, "t_in")
    _f32(W, "W", (N_out, N_in))
    _f32(t_out, "t_out", (B, N_out))
    _f32(g_t_out, "g_t_out", (B, N_out))
    _f32(g_W, "g_W", (N_out, N_in))
    if g_t_in is not None:
        _f32(g_t_in, "g_t_in", (B, N_in))
    _check(load().dstd_exact_bwd(_ptr(t_in), _ptr(W), _ptr(t_out), _ptr(g_t_out), B, N_in, N_out, ctypes.byref(p),
                                 _ptr(g_t_in) if g_t_in is not None else None, _ptr(g_W), _ptr(workspace),
                                 workspace.numel() * workspace.element_size(), _stream(stream)), "dstd_exact_bwd")


def set_pair_policy(policy):
    """Forward contraction scheduling: 0 cost model (default), 1 SM pairs
    wherever they apply, 2 single CTAs only. Returns the previous policy."""
    r = load().dstd_set_pair_policy(int(policy))
    if r < 0:
        raise DstdError(r, "dstd_set_pair_policy")
    return r


def conv_set_chunk_images(max_images):
    """Cap the images per chunk of the implicit-GEMM conv layers (0 = from
    the scratch budget). Returns the previous cap; query the workspace size
    again afterwards."""
    return int(load().dstd_conv_set_chunk_images(int(max_images)))


def conv_set_operand_policy(policy):
    """Operand of the implicit-GEMM conv forward and dW: 0 by layer shape,
    1 generated on chip, 2 the binned input written out and read through
    TMA. Returns the previous policy; query the workspace size again."""
    return int(load().dstd_conv_set_operand_policy(int(policy)))


def timing_collect():
    """Add the last replay of a graph captured with timing on to the totals."""
    _check(load().dstd_timing_collect(), "dstd_timing_collect")


def timing_read():
    """{kernel kind: (total ms, launches)} accumulated since timing_enable."""
    lib = load()
    out = {}
    for k in range(lib.dstd_kernel_kind_count()):
        ms = _F()
        n = _I64()
        _check(lib.dstd_timing_read(k, ctypes.byref(ms), ctypes.byref(n)), "dstd_timing_read")
        out[lib.dstd_kernel_kind_name(k).decode()] = (ms.value, n.value)
    return out


def selftest_wait_timeout(timeout_us, stream=None):
    """Launch the bounded-wait self-test (see include/dstd.h)."""
    _check(load().dstd_selftest_wait_timeout(int(timeout_us), _stream(stream)), "dstd_selftest_wait_timeout")
