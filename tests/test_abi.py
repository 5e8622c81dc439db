"""CPU checks of the C-ABI: the library builds for sm_103a, loads, exports every
function include/dstd.h declares, and rejects bad arguments on the host
before anything is launched (no GPU needed)."""

import ctypes
import math
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="nvcc not available")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_14672_gb300 import build, dstd
    build.build()
    return dstd.load()


def declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(dstd_\w+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 13
    for n in names:
        assert hasattr(lib, n), n
    from paper_2607_14672_gb300 import dstd
    assert set(dstd.EXPORTS) == names


def test_version_and_errors(lib):
    from paper_2607_14672_gb300 import dstd
    assert dstd.version() == 100
    for code, msg in dstd.ERRORS.items():
        assert dstd.error_string(code) == msg
    assert dstd.error_string(-99) == "unknown error code"


def _layer(M=32, **kw):
    from paper_2607_14672_gb300 import dstd
    L = dict(tau_v=0.5, tau_I=0.25, v_th=1.0, t_first=0.0, t_end=1.2, M=M, t_offset=0.0)
    L.update(kw)
    return dstd.params(L, 1.0 / 8)


def test_size_queries(lib):
    from paper_2607_14672_gb300 import dstd
    p = _layer()
    # q, s, vdot: 320 bytes each at 256-byte aligned offsets 0, 512, 1024
    assert dstd.dense_saved_bytes(8, 10) == 2 * 512 + 8 * 10 * 4
    for m in ("f32", "x3", "bf16"):
        assert dstd.dense_workspace_bytes(256, 784, 800, p, m) > 0
    # the three-product split carries two copies of each operand
    assert dstd.dense_workspace_bytes(256, 784, 800, p, "x3") > dstd.dense_workspace_bytes(256, 784, 800, p, "bf16")
    # invalid constants -> 0
    for bad in (dict(tau_v=-1.0), dict(tau_I=0.0), dict(v_th=0.0), dict(t_end=-1.0), dict(M=0),
                dict(t_offset=0.5), dict(t_offset=-0.02), dict(tau_v=math.nan)):
        assert dstd.dense_workspace_bytes(8, 16, 16, _layer(**bad), "f32") == 0, bad
    # infinite time constants are valid
    assert dstd.dense_workspace_bytes(8, 16, 16, _layer(tau_v=math.inf, tau_I=math.inf), "f32") > 0
    # tensor-core modes take M <= 128; the fp32 mode up to 256; beyond that nothing
    assert dstd.dense_workspace_bytes(8, 16, 16, _layer(M=200), "x3") == 0
    assert dstd.dense_workspace_bytes(8, 16, 16, _layer(M=200), "f32") > 0
    assert dstd.dense_workspace_bytes(8, 16, 16, _layer(M=300), "f32") == 0
    assert dstd.dense_workspace_bytes(0, 16, 16, p, "f32") == 0
    assert dstd.dense_workspace_bytes(8, 0, 16, p, "f32") == 0
    # the conv operand policy: writing the binned input out (2) puts S
    # [images, H, W, Mp, C_in] bf16 in the workspace of a 128-channel layer
    # in place of the 8-byte records
    assert dstd.conv_set_operand_policy(-1) == 0 and dstd.conv_set_operand_policy(3) == 0
    assert dstd.conv_set_operand_policy(1) == 0
    pm = _layer(M=64)
    try:
        w_gen = dstd.conv_workspace_bytes(2, 8, 8, 128, 128, 3, 1, 1, pm, "bf16")
        assert dstd.conv_set_operand_policy(2) == 1
        w_tma = dstd.conv_workspace_bytes(2, 8, 8, 128, 128, 3, 1, 1, pm, "bf16")
        S, rec = 2 * 8 * 8 * 64 * 128 * 2, 2 * 8 * 8 * 128 * 8
        assert abs((w_tma - w_gen) - (S - rec)) <= 2 * 256
    finally:
        dstd.conv_set_operand_policy(0)


def test_null_and_bad_arguments_rejected_on_host(lib):
    from paper_2607_14672_gb300 import dstd
    p = ctypes.byref(_layer())
    one = ctypes.c_void_p(256)
    assert lib.dstd_dense_fwd(None, one, 8, 16, 16, p, 0, one, one, None, one, 1 << 20, None) == -1
    assert lib.dstd_dense_fwd(one, one, 0, 16, 16, p, 0, one, one, None, one, 1 << 20, None) == -1
    assert lib.dstd_dense_fwd(one, one, 8, 16, 16, None, 0, one, one, None, one, 1 << 20, None) == -1
    assert lib.dstd_dense_fwd(one, one, 8, 16, 16, p, 7, one, one, None, one, 1 << 20, None) == -1
    # misaligned pointer
    odd = ctypes.c_void_p(258)
    assert lib.dstd_dense_fwd(odd, one, 8, 16, 16, p, 0, one, one, None, one, 1 << 20, None) == -1
    # workspace too small
    assert lib.dstd_dense_fwd(one, one, 8, 16, 16, p, 1, one, one, None, one, 16, None) == -3
    assert lib.dstd_dense_bwd(one, one, one, one, one, 8, 16, 16, p, 1, None, None, one, 1 << 20, None) == -1
    assert lib.dstd_dense_bwd(one, one, one, one, one, 8, 16, 16, p, 1, None, one, one, 16, None) == -3
    assert lib.dstd_binning(None, 8, 16, p, one, None, None) == -1
    assert lib.dstd_scan_solve(one, 8, 16, p, None, None, None, None, None) == -1
    assert lib.dstd_dense_what(one, one, 8, 16, 16, p, 0, None, one, 1 << 20, None) == -1
    assert lib.dstd_ce_loss(one, one, 8, 10, ctypes.c_float(0.0), ctypes.c_float(1.0), one, one, None) == -1
    assert lib.dstd_sum_t_loss(one, 0, one, one, None) == -1
    assert lib.dstd_adamw(one, one, one, one, 10, ctypes.c_float(1e-3), ctypes.c_float(1.5), ctypes.c_float(0.9),
                          ctypes.c_float(1e-8), ctypes.c_float(0.0), 1, None) == -1
    assert lib.dstd_adamw(one, one, one, one, 10, ctypes.c_float(1e-3), ctypes.c_float(0.9), ctypes.c_float(0.9),
                          ctypes.c_float(1e-8), ctypes.c_float(0.0), 0, None) == -1
    # contraction scheduling policy: 0, 1, 2 valid (previous returned), anything else rejected
    assert lib.dstd_set_pair_policy(3) == -1 and lib.dstd_set_pair_policy(-1) == -1
    # multi-spike layers: spike counts 1..8, tensor-core modes only, checked before any device call
    ms_args = lambda Fi, Fo, math: (one, one, 8, 16, 16, Fi, Fo, p, math, one, one, one, 1 << 30, None)
    assert lib.dstd_dense_fwd_ms(*ms_args(0, 2, 1)) == -1
    assert lib.dstd_dense_fwd_ms(*ms_args(2, 0, 1)) == -1
    assert lib.dstd_dense_fwd_ms(*ms_args(9, 2, 1)) == -2
    assert lib.dstd_dense_fwd_ms(*ms_args(2, 9, 1)) == -2
    assert lib.dstd_dense_fwd_ms(*ms_args(2, 2, 0)) == -2                     # fp32 CUDA-core mode
    assert lib.dstd_dense_bwd_ms(one, one, one, one, one, 8, 16, 16, 2, 9, p, 1, None, one, one, 1 << 30,
                                 None) == -2
    assert lib.dstd_dense_bwd_ms(one, one, one, one, one, 8, 16, 16, 2, 2, p, 1, None, None, one, 1 << 30,
                                 None) == -1                                   # no g_W
    assert lib.dstd_ms_saved_bytes(8, 16, 0) == 0 and lib.dstd_ms_saved_bytes(8, 16, 9) == 0
    assert lib.dstd_ms_saved_bytes(8, 16, 3) >= 8 * 16 * 3 * 12
    assert lib.dstd_ms_workspace_bytes(8, 16, 16, 2, 2, p, 0) == 0
    assert lib.dstd_ms_workspace_bytes(8, 16, 16, 2, 2, p, 1) > 0
    # skip-and-delay channel concatenation and its adjoint
    assert lib.dstd_concat_channels(None, 4, ctypes.c_float(0.2), one, 4, 10, one, None) == -1
    assert lib.dstd_concat_channels(one, 0, ctypes.c_float(0.2), one, 4, 10, one, None) == -1
    assert lib.dstd_concat_channels(one, 4, ctypes.c_float(float("inf")), one, 4, 10, one, None) == -1
    assert lib.dstd_split_channels(one, 4, 4, 10, None, 0, None, 0, None) == -1
    assert lib.dstd_split_channels(one, 4, 4, 0, one, 0, one, 0, None) == -1
    assert lib.dstd_set_pair_policy(2) == 0 and lib.dstd_set_pair_policy(0) == 2
    assert lib.dstd_conv_set_chunk_images(-1) == 0
    assert lib.dstd_conv_set_chunk_images(3) == 0 and lib.dstd_conv_set_chunk_images(0) == 3
    # multi-tensor AdamW: tensor count, null step buffer, misaligned step buffer, empty tensor, bad beta
    ptrs = (ctypes.c_void_p * 33)(*([256] * 33))
    ns = (ctypes.c_int64 * 33)(*([10] * 33))
    hyper = (ctypes.c_float(1e-3), ctypes.c_float(0.9), ctypes.c_float(0.999), ctypes.c_float(1e-8),
             ctypes.c_float(0.0))
    assert lib.dstd_adamw_multi(0, ptrs, ptrs, ptrs, ptrs, ns, *hyper, one, None, None) == -1
    assert lib.dstd_adamw_multi(33, ptrs, ptrs, ptrs, ptrs, ns, *hyper, one, None, None) == -1
    assert lib.dstd_adamw_multi(2, ptrs, ptrs, ptrs, ptrs, ns, *hyper, None, None, None) == -1
    assert lib.dstd_adamw_multi(2, ptrs, ptrs, ptrs, ptrs, ns, *hyper, ctypes.c_void_p(260), None, None) == -1
    n0 = (ctypes.c_int64 * 2)(10, 0)
    assert lib.dstd_adamw_multi(2, ptrs, ptrs, ptrs, ptrs, n0, *hyper, one, None, None) == -1
    assert lib.dstd_adamw_multi(2, ptrs, ptrs, ptrs, ptrs, ns, ctypes.c_float(1e-3), ctypes.c_float(1.0),
                                ctypes.c_float(0.999), ctypes.c_float(1e-8), ctypes.c_float(0.0), one, None,
                                None) == -1
