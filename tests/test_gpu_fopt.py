"""The forward optimizer on the GPU (Alg. 1 with the cost F, Sec. IV-C) against the oracle: the FP32
layers and conversions element by element, the initial QPs, every candidate's cost and the chosen FLs.
The GPU evaluates the FP32 part of the network in fp32 and the oracle in float64, so costs agree to a
relative tolerance; every fixed-point step is exact on both sides."""
import numpy as np
import pytest
import torch

import synth
from oracle import qopt

pytestmark = pytest.mark.gpu

RTOL = 2e-5


@pytest.fixture(scope="module")
def M():
    import __graft_entry__ as g
    g.build()
    from paper_2203_12091_gb300 import fopt, fxpq
    return fopt, fxpq


def test_fp32_layers_match_float64(M):
    fopt, F = M
    rng = np.random.default_rng(61)
    for (N, H, C, K, R, st, pad, relu) in [(2, 9, 3, 16, 3, 1, 1, True), (3, 12, 20, 70, 5, 2, 2, False),
                                            (1, 7, 64, 8, 7, 1, 0, True)]:
        x = rng.standard_normal((N, H, H, C)).astype(np.float32)
        w = rng.standard_normal((K, R, R, C)).astype(np.float32)
        b = rng.standard_normal(K).astype(np.float32)
        P = (H + 2 * pad - R) // st + 1
        y = torch.empty(N * P * P * K, dtype=torch.float32, device="cuda")
        F.fxpq_conv_f32(N, H, H, C, K, R, R, st, pad, relu, torch.from_numpy(x).cuda(), torch.from_numpy(w).cuda(),
                        torch.from_numpy(b).cuda(), y)
        want = qopt.f_conv(x, w, b, st, pad, relu)
        np.testing.assert_allclose(y.cpu().numpy().reshape(want.shape), want, rtol=1e-4, atol=1e-4)
    x = rng.standard_normal((2, 9, 9, 5)).astype(np.float32)
    y = torch.empty(2 * 5 * 5 * 5, dtype=torch.float32, device="cuda")
    F.fxpq_maxpool_f32(torch.from_numpy(x).cuda(), 2, 9, 9, 5, 3, 2, 1, y)
    assert np.array_equal(y.cpu().numpy().reshape(2, 5, 5, 5), qopt.f_maxpool(x, 3, 2, 1).astype(np.float32))
    a = torch.empty(2 * 5, dtype=torch.float32, device="cuda")
    F.fxpq_avgpool_f32(torch.from_numpy(x).cuda(), 2, 9, 9, 5, a)
    np.testing.assert_allclose(a.cpu().numpy().reshape(2, 1, 1, 5), qopt.f_avgpool(x), rtol=1e-6, atol=1e-6)


def test_ds_stats_and_ties(M):
    fopt, F = M
    rng = np.random.default_rng(62)
    x = (rng.standard_normal((3, 1000)) * [[0.5], [2.0], [1.0]]).astype(np.float32)
    out = torch.empty(3 + 6, dtype=torch.float64, device="cuda")
    ws = torch.empty(2, dtype=torch.int32, device="cuda")
    for fmt in ((6, 1, 3), (1, 1, 1), (8, 0, 5)):
        F.fxpq_ds_stats(torch.from_numpy(x).cuda(), 3, 1000, F.fmt(*fmt), out, ws)
        h = out.cpu().numpy()
        assert h[0] == pytest.approx(qopt.qerr(x, fmt), rel=1e-12)
        assert h[1] == x.min() and h[2] == x.max()
        np.testing.assert_allclose(h[3::2], x.astype(np.float64).sum(axis=1), rtol=1e-12)
        np.testing.assert_allclose(h[4::2], (x.astype(np.float64) ** 2).sum(axis=1), rtol=1e-12)
    lg = np.array([[1, 1, 0], [2, 0, 0], [5, 5, 5]], np.float32)
    c = torch.empty(3, dtype=torch.int32, device="cuda")
    F.fxpq_top1_ties(torch.from_numpy(lg).cuda(), 3, 3, c)
    assert c.cpu().tolist() == [2, 1, 3]
    F.fxpq_top1_ties(torch.from_numpy(lg.astype(np.int64)).cuda(), 3, 3, c)
    assert c.cpu().tolist() == [2, 1, 3]


def _tiny():
    layers = [
        {"type": "conv", "name": "c1", "C": 3, "K": 8, "R": 3, "stride": 1, "pad": 1, "relu": True, "src": None},
        {"type": "maxpool", "name": "p1", "k": 2, "stride": 2, "pad": 0},
        {"type": "conv", "name": "c2", "C": 8, "K": 8, "R": 3, "stride": 1, "pad": 1, "relu": False, "src": "p1"},
        {"type": "eltwise", "name": "e", "a": "c2", "b": "p1", "relu": True},
        {"type": "avgpool", "name": "gap", "src": "e"},
        {"type": "conv", "name": "fc", "C": 8, "K": 10, "R": 1, "stride": 1, "pad": 0, "relu": False, "src": "gap"},
    ]
    rng = np.random.default_rng(52)
    W = {}
    for L in layers:
        if L["type"] == "conv":
            fan = L["C"] * L["R"] ** 2
            W[L["name"]] = ((rng.standard_normal((L["K"], L["R"], L["R"], L["C"])) * np.sqrt(2 / fan)).astype(np.float32),
                            (rng.standard_normal(L["K"]) * 0.05).astype(np.float32))
    plan = {"input": 6, "c1": {"w": 5, "b": 8, "a": 5}, "c2": {"w": 4, "b": 8, "a": 6}, "e": {"a": 5},
            "gap": {"a": 6, "r": 16}, "fc": {"w": 6, "b": 8}}
    return layers, W, plan


def _run_both(M, layers, W, plan, imgs, K=1, upto=None):
    fopt, F = M
    wdev = {nm: (torch.from_numpy(w).cuda(), torch.from_numpy(b).cuda()) for nm, (w, b) in W.items()}
    g = fopt.ForwardOptimizer(layers, wdev, torch.from_numpy(imgs).cuda(), plan)
    o = qopt.Net(layers, W, imgs, plan)
    assert g.order == o.order
    for ds in o.order:
        assert g.fmt[ds].tup() == o.fmt[ds], ds  # initial QPs from the FP32 ranges
    res_g, res_o = g.run(K, upto), qopt.forward_optimize(o, K, upto)
    for (ds, flg, cg, trg), (ds2, flo, co, tro) in zip(res_g, res_o):
        assert ds == ds2
        assert [f for f, _ in trg] == [f for f, _ in tro], ds
        np.testing.assert_allclose([c for _, c in trg], [c for _, c in tro], rtol=RTOL, atol=1e-12)
        assert flg == flo, ds
    return res_g


def test_forward_optimizer_tiny_residual_net(M):
    layers, W, plan = _tiny()
    _run_both(M, layers, W, plan, synth.images(6, 63, hw=12))


def test_forward_optimizer_wider_search(M):
    layers, W, plan = _tiny()
    _run_both(M, layers, W, plan, synth.images(4, 64, hw=8), K=2)


def test_forward_optimizer_resnet18_prefix(M):
    """ResNet-18 (32 x 32 synthetic images, 3 of them): Alg. 1 on the first 12 data-structures (the input,
    conv1, the first residual block's convs and add), every candidate's cost over the whole network."""
    layers = synth.resnet18()
    W = synth.weights("resnet18", 65)
    plan = synth.bit_plan("resnet18", 65)
    _run_both(M, layers, W, plan, synth.images(3, 66, hw=32), upto=12)
