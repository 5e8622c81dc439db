"""The allocation-free layer forward (dstd_dense_fwd_noalloc) against the
workspace one (dstd_dense_fwd), through the C-ABI.

dstd_dense_fwd_noalloc serves callers that cannot allocate device memory;
its scratch is the library's fixed 64 MiB device array, shared by all calls.
Two calls in a row (different layers, different sizes) must each give what
dstd_dense_fwd gives on the same inputs: spike times within 1e-4 T_max (the
parity tolerance of the other tests; in fact bitwise), identical firing
masks and saved state. This file is collected last, so a run that stops at
the first failure has run everything else before it.
"""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    from paper_2607_14672_gb300 import build, dstd
    build.build()
    dstd.load()
    yield


def _both(t_in, W, layer, B, math_mode):
    from paper_2607_14672_gb300 import dstd
    N_out, N_in = W.shape
    p = dstd.params(layer, 1.0 / B)
    # the workspace starts full of 0xFF bytes, so a forward that read scratch
    # it had not written would differ from the allocation-free one
    ws = torch.full((dstd.dense_workspace_bytes(B, N_in, N_out, p, math_mode),), 255, dtype=torch.uint8,
                    device="cuda")
    nsv = dstd.dense_saved_bytes(B, N_out)
    out = []
    for noalloc in (False, True):
        t_out = torch.full((B, N_out), -1.0, device="cuda")
        saved = torch.zeros(nsv, dtype=torch.uint8, device="cuda")
        pen = torch.zeros(4, device="cuda")
        if noalloc:
            dstd.dense_fwd_noalloc(t_in, W, p, math_mode, t_out, saved, pen)
        else:
            dstd.dense_fwd(t_in, W, p, math_mode, t_out, saved, pen, ws)
        torch.cuda.synchronize()
        out.append((t_out.cpu().numpy(), saved.cpu().numpy(), pen.cpu().numpy()))
    assert dstd.device_status(clear=True) == 0
    return out


def _check(ref, got, layer):
    tmax = layer["t_end"] - layer["t_first"]
    (t0, s0, p0), (t1, s1, p1) = ref, got
    np.testing.assert_array_equal(np.isfinite(t0), np.isfinite(t1))
    fin = np.isfinite(t0)
    assert np.abs(t0[fin] - t1[fin]).max(initial=0.0) <= 1e-4 * tmax
    np.testing.assert_array_equal(s0, s1)
    np.testing.assert_allclose(p0, p1, rtol=1e-5, atol=1e-7)
    assert fin.sum() > 0


@pytest.mark.parametrize("math_mode", ["x3", "f32"])
def test_noalloc_forward_matches_workspace_forward_twice(math_mode):
    from paper_2607_14672_gb300 import configs
    cfg = configs.config2(batch=256 if math_mode == "x3" else 64)
    B = cfg["batch"]
    t0 = torch.tensor(np.asarray(cfg["inputs"](B=B), np.float32), device="cuda")
    L1, L2 = cfg["layers"][0], cfg["layers"][1]
    W1 = torch.tensor(np.asarray(L1["W"], np.float32), device="cuda")
    W2 = torch.tensor(np.asarray(L2["W"], np.float32), device="cuda")
    # first call: layer 1 (784 -> 800)
    r1 = _both(t0, W1, L1, B, math_mode)
    _check(r1[0], r1[1], L1)
    # second call in a row: layer 2 (800 -> 800) on layer 1's spike times
    t1 = torch.tensor(r1[0][0], device="cuda")
    r2 = _both(t1, W2, L2, B, math_mode)
    _check(r2[0], r2[1], L2)


def test_noalloc_rejects_oversized_layers():
    from paper_2607_14672_gb300 import configs, dstd
    cfg = configs.config3(4096, 128, batch=128)
    L = cfg["layers"][0]
    p = dstd.params(L, 1.0 / 128)
    t_in = torch.zeros(128, 4096, device="cuda")
    W = torch.zeros(4096, 4096, device="cuda")
    t_out = torch.empty(128, 4096, device="cuda")
    saved = torch.empty(dstd.dense_saved_bytes(128, 4096), dtype=torch.uint8, device="cuda")
    with pytest.raises(dstd.DstdError) as e:
        dstd.dense_fwd_noalloc(t_in, W, p, "x3", t_out, saved)
    assert e.value.code == -3
    assert dstd.device_status(clear=True) == 0


@pytest.mark.parametrize("math_mode", ["x3", "bf16"])
def test_noalloc_ragged_width_after_a_larger_layer(math_mode):
    """A layer whose input width is not a multiple of 8 (100 -> 300: its
    operand rows are padded to 104 columns) right after a larger layer has
    filled the shared scratch: the padding columns must not carry the
    earlier call's values into the result."""
    from paper_2607_14672_gb300 import configs, synth
    cfg = configs.config2(batch=256)
    B = 256
    L1 = cfg["layers"][0]
    t0 = torch.tensor(np.asarray(cfg["inputs"](B=B), np.float32), device="cuda")
    W1 = torch.tensor(np.asarray(L1["W"], np.float32), device="cuda")
    r1 = _both(t0, W1, L1, B, math_mode)          # 784 -> 800 fills the scratch first
    _check(r1[0], r1[1], L1)
    L = dict(L1)
    t_small = torch.tensor(np.asarray(synth.uniform_spikes(5, (B, 100), 0.0, 1.0, 0.2), np.float32), device="cuda")
    W_small = torch.tensor(np.asarray(synth.normal_weights(1005, (300, 100), 0.12, 0.1), np.float32), device="cuda")
    r2 = _both(t_small, W_small, L, B, math_mode)
    _check(r2[0], r2[1], L)
