"""The paper's architectures as the workload definitions build them
(Tab. architectures, Fig. skip_connection, App. C.2), checked on the host."""

import numpy as np

from paper_2607_14672_gb300 import configs


def _conv_specs(cfg):
    return [(L["W"].shape[0], L["W"].shape[1], L["W"].shape[2], L["stride"], L["pad"], L.get("skip"))
            for L in cfg["layers"] if L["kind"] == "conv"]


def test_syn_snn9_architecture():
    # C(N,3,1)-C(N,3,1)-C(N,3,1)-C(N,3,2)-C(2N,3,1)-C(2N,3,1)-C(2N,3,2)-C(2N,5,1)-10
    N = 8
    cfg = configs.syn_snn9(N=N, batch=2, M=20, mus=(0.0,) * 9)
    specs = _conv_specs(cfg)
    assert [s[0] for s in specs] == [N, N, N, N, 2 * N, 2 * N, 2 * N, 2 * N]
    assert [s[2] for s in specs] == [3] * 7 + [5]
    assert [s[3] for s in specs] == [1, 1, 1, 2, 1, 1, 2, 1]
    assert all(s[4] == s[2] // 2 and s[5] is None for s in specs)
    assert specs[0][1] == 6                                   # doubled colour input
    assert [s[1] for s in specs[1:]] == [s[0] for s in specs[:-1]]
    assert cfg["shapes"][-2] == (2 * N, 8, 8)                 # 32 -> 16 -> 8
    assert cfg["layers"][-1]["W"].shape == (10, 2 * N * 8 * 8)
    assert len(cfg["layers"]) == 9


def test_doubled_input_channels():
    # App. C.2: x_{k+3} = 1 - x_k, so with t = tau_in (1 - x) the two halves add to tau_in
    cfg = configs.syn_snn9(N=4, batch=3, mus=(0.0,) * 9)
    t = cfg["inputs"]()
    assert t.shape == (3, 6, 32, 32)
    np.testing.assert_allclose(t[:, :3] + t[:, 3:], configs.SYNFIRE["tau_in"], atol=1e-15)
    assert np.isfinite(t).all() and (t >= 0).all() and (t <= 1).all()


def test_syn_snn20_architecture():
    # C(N,K,S)-SD2(N)-SD1(N)-SD2(2N)-SD1(2N)-SD2(4N)-SD1(4N)-10: 1 + 6 x 3 convs + readout
    N = 4
    cfg = configs.syn_snn20(N=N, batch=2, M=20, mus=(0.0,) * 20)
    specs = _conv_specs(cfg)
    assert len(specs) == 19 and len(cfg["layers"]) == 20
    delay = 2 * configs.SYNFIRE["tau_shift"]
    skip_layers = [l for l, s in enumerate(specs) if s[5] is not None]
    assert skip_layers == [3, 6, 9, 12, 15, 18]
    widths = [N, N, 2 * N, 2 * N, 4 * N, 4 * N]
    for b, l in enumerate(skip_layers):
        src, d = specs[l][5]
        assert src == l - 3 and d == delay                    # the block's input, delayed 2 tau_shift
        w = widths[b]
        sd1 = b % 2 == 1
        # first two layers of the block: w channels, stride 1
        assert specs[l - 2][0] == w and specs[l - 1][0] == w
        assert specs[l - 2][3] == 1 and specs[l - 1][3] == 1
        # third: reads the block input and the second layer's output along channels
        assert specs[l][1] == specs[src][0] + specs[l - 1][0]
        assert specs[l][0] == (2 * w if sd1 else w) and specs[l][3] == (2 if sd1 else 1)
    assert cfg["shapes"][-2] == (8 * N, 4, 4)                 # 28 -> 14 -> 7 -> 4
    assert cfg["layers"][-1]["W"].shape == (10, 8 * N * 16)
    # synfire windows advance by tau_shift per layer
    firsts = [L["t_first"] for L in cfg["layers"]]
    np.testing.assert_allclose(np.diff(firsts), configs.SYNFIRE["tau_shift"])
