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


def test_ds_stats_batch_and_ties(M):
    """Statistics records (Eq. DSB_QE's L, the range ends, per-sample mean and sum of squared deviations)
    against float64 numpy, several items in one batch, one of them past one work unit per sample; a
    data-structure with a large mean and a small spread keeps its deviation (no one-pass cancellation)."""
    fopt, F = M
    rng = np.random.default_rng(62)
    xs = [(rng.standard_normal((3, 1000)) * [[0.5], [2.0], [1.0]]).astype(np.float32),
          (rng.standard_normal((2, 70000)) * 0.001 + 1000.0).astype(np.float32),
          rng.standard_normal((1, 5)).astype(np.float32)]
    for fmt in ((6, 1, 3), (1, 1, 1), (8, 0, 5)):
        outs = [torch.empty(3 + 2 * x.shape[0], dtype=torch.float64, device="cuda") for x in xs]
        F.fxpq_ds_stats_batch([(torch.from_numpy(x).cuda().reshape(-1), x.shape[0], x.shape[1], F.fmt(*fmt), o)
                               for x, o in zip(xs, outs)])
        for x, o in zip(xs, outs):
            h = o.cpu().numpy()
            x64 = x.astype(np.float64)
            assert h[0] == pytest.approx(qopt.qerr(x, fmt), rel=1e-12)
            assert h[1] == x.min() and h[2] == x.max()
            np.testing.assert_allclose(h[3::2], x64.mean(axis=1), rtol=1e-14)
            np.testing.assert_allclose(h[4::2], ((x64 - x64.mean(axis=1, keepdims=True)) ** 2).sum(axis=1), rtol=1e-9)
    lg = np.array([[1, 1, 0], [2, 0, 0], [5, 5, 5]], np.float32)
    c = torch.empty(3, dtype=torch.int32, device="cuda")
    F.fxpq_top1_ties(torch.from_numpy(lg).cuda(), 3, 3, c)
    assert c.cpu().tolist() == [2, 1, 3]
    F.fxpq_top1_ties(torch.from_numpy(lg.astype(np.int64)).cuda(), 3, 3, c)
    assert c.cpu().tolist() == [2, 1, 3]


def test_fopt_cost_from_records(M):
    """fxpq_fopt_cost on hand-made records: E by Eq. importance / Eq. CPB_QE per layer, UnClass and
    MisPred by their equations, two candidates with their own records and ties."""
    fopt, F = M
    # candidate 0: layer 0 = {a: 2 samples, nu 4}, {w: 1 sample, nu 6}; layer 1 = {w: nu 3 with R = 0}
    rec0 = [[0.5, -1.0, 3.0, 0.2, 1.0, 0.1, 4.0], [0.25, -2.0, 2.0, 0.0, 6.0], [0.1, 1.0, 1.0, 1.0, 0.0]]
    rec1 = [[1.5, -1.0, 1.0, 0.0, 0.25, 0.0, 1.0], [0.0, -2.0, 2.0, 0.0, 1.5], [0.3, 0.0, 2.0, 1.0, 3.0]]
    layout = [(0, 4, 2, 0), (7, 6, 1, 0), (12, 3, 1, 1)]
    stats = torch.tensor(sum(rec0, []) + sum(rec1, []), dtype=torch.float64, device="cuda")
    ties = torch.tensor([1, 2, 1, 3, 1, 1, 1, 1], dtype=torch.int32, device="cuda")
    cost = torch.empty(8, dtype=torch.float64, device="cuda")
    F.fxpq_fopt_cost(stats, 17, layout, ties, 4, 5, 2, cost)
    got = cost.cpu().numpy().reshape(2, 4)
    for c, recs in enumerate((rec0, rec1)):
        E = 0.0
        for layer in (0, 1):
            ts = [(r, nu, ns) for r, (o, nu, ns, ly) in zip(recs, layout) if ly == layer]
            sig = [sum(np.sqrt(r[4 + 2 * s_] / nu) for s_ in range(ns)) / ns for r, nu, ns in ts]
            den = sum(sg * nu for sg, (r, nu, ns) in zip(sig, ts))
            for sg, (r, nu, ns) in zip(sig, ts):
                if den > 0 and r[2] > r[1]:
                    E += sg * nu / den * r[0] / (r[2] - r[1])
        t = ties.cpu().numpy()[4 * c:4 * c + 4]
        uc, mp = np.mean(t > 1), (t - 1).sum() / (4 * 5)
        np.testing.assert_allclose(got[c], [E + uc + mp, E, uc, mp], rtol=1e-14)


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
