"""Network parity on the GPU: calibration (formats chosen by the FL search in the forward
optimizer's order) and the integer-only forward through fxpq_net_forward, against the oracle.

The forward runs on the full batch of each workload (the launch configuration the bench times);
the oracle recomputes sampled images of that batch one by one."""
import numpy as np
import pytest
import torch

import synth
from oracle import net as onet

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def NET():
    import __graft_entry__ as g
    g.build()
    from paper_2203_12091_gb300 import net
    return net


def fmts_equal(gpu_fmts, ora_fmts):
    for nm, d in ora_fmts.items():
        if nm == "input":
            assert gpu_fmts["input"]["a"].tup() == tuple(d), nm
            continue
        for key, f in d.items():
            assert gpu_fmts[nm][key].tup() == tuple(f), (nm, key)


def _tiny():
    L = [
        {"type": "conv", "name": "c1", "C": 3, "K": 16, "R": 3, "stride": 2, "pad": 1, "relu": True, "src": None},
        {"type": "maxpool", "name": "p1", "k": 3, "stride": 2, "pad": 1},
        {"type": "conv", "name": "a", "C": 16, "K": 16, "R": 3, "stride": 1, "pad": 1, "relu": True, "src": "p1"},
        {"type": "conv", "name": "b", "C": 16, "K": 16, "R": 3, "stride": 1, "pad": 1, "relu": False, "src": "a"},
        {"type": "eltwise", "name": "e", "a": "b", "b": "p1", "relu": True},
        {"type": "avgpool", "name": "gap", "src": "e"},
        {"type": "conv", "name": "fc", "C": 16, "K": 24, "R": 1, "stride": 1, "pad": 0, "relu": False, "src": "gap"},
    ]
    plan = {"input": 7, "c1": {"w": 6, "b": 16, "a": 8}, "a": {"w": 5, "b": 16, "a": 6}, "b": {"w": 8, "b": 16, "a": 7},
            "e": {"a": 5}, "gap": {"a": 8, "r": 16}, "fc": {"w": 16, "b": 16}}
    return L, plan


def test_tiny_residual_net(NET):
    L, plan = _tiny()
    rng = np.random.default_rng(1)
    W = {}
    for l in L:
        if l["type"] == "conv":
            fan = l["C"] * l["R"] ** 2
            W[l["name"]] = ((rng.standard_normal((l["K"], l["R"], l["R"], l["C"])) * np.sqrt(2 / fan)).astype(np.float32),
                            (rng.standard_normal(l["K"]) * 0.01).astype(np.float32))
    imgs = synth.images(6, 2, hw=28)
    q = NET.build_qnet(L, W, torch.from_numpy(imgs[:4]).cuda(), plan)
    fm, qp = onet.calibrate(L, W, imgs[:4], plan)
    fmts_equal(q.fmts, fm)
    logits, s = q.forward(torch.from_numpy(imgs).cuda())
    want, ws = onet.forward(L, fm, qp, imgs)
    assert s == ws and np.array_equal(logits.cpu().numpy(), want)
    # per-layer codes of the op-by-op path agree too
    env = q.trace(torch.from_numpy(imgs).cuda())
    oenv = onet.forward_trace(L, fm, qp, imgs)
    from paper_2203_12091_gb300 import fxpq as F
    for l in L[:-1]:
        t, f = env[l["name"]]
        H, _, Cp = q.shapes[l["name"]]
        got = F.codes_to_int(t.cpu(), f, (6, H, H, Cp)).numpy()
        assert np.array_equal(got[..., : oenv[l["name"]][0].shape[-1]], oenv[l["name"]][0]), l["name"]


def _workload(NET, arch, batch, seed, plan_seed=None, calib=8, sample=(0, -1), pack=False):
    L = synth.ARCHS[arch]()
    W = synth.weights(arch, seed)
    plan = synth.bit_plan(arch, seed if plan_seed is None else plan_seed)
    bn = synth.bn_params(arch, seed + 100)
    imgs = synth.images(batch, seed)
    dimgs = torch.from_numpy(imgs).cuda()
    q = NET.build_qnet(L, W, dimgs[:calib], plan, bn_np=bn, pack_weights=pack)
    if pack:
        assert q.qp, "no layer took packed weights"
    fm, qp = onet.calibrate(L, W, imgs[:calib], plan, bn)
    fmts_equal(q.fmts, fm)
    logits, s = q.forward(dimgs)
    torch.cuda.synchronize()
    got = logits.cpu().numpy()
    idx = [i % batch for i in sample]
    want, ws = onet.forward(L, fm, qp, imgs[idx])
    assert s == ws
    assert np.array_equal(got[idx], want)
    from paper_2203_12091_gb300 import fxpq as F
    assert F.fxpq_get_device_status() == 0
    return got


def test_alexnet_batch256(NET):
    _workload(NET, "alexnet", 256, 5)


def test_alexnet_batch256_packed_fc_weights(NET):
    """The same workload with its three FC layers' 8-bit weights read as packed 8-bit planes
    (Sec. V-E.2) by the contraction, calibration included: formats and logits equal the oracle's."""
    _workload(NET, "alexnet", 256, 5, pack=True)


def test_resnet18_batch128(NET):
    _workload(NET, "resnet18", 128, 6)


def test_resnet18_bn_batch128(NET):
    """ResNet-18 with its BN layers kept as Scale layers (bias-free convs, aleph1 / aleph2 applied in the
    conv epilogue before ReLU), the paper's own form of the network."""
    _workload(NET, "resnet18_bn", 128, 6)


def test_bn_to_scale_bit_exact(NET):
    """fxpq_bn_to_scale against the oracle's fp32 formula, bit for bit (every step correctly rounded)."""
    from oracle import bn_to_scale
    from paper_2203_12091_gb300 import fxpq as F
    rng = np.random.default_rng(31)
    n = 10007
    g = rng.uniform(-2, 2, n).astype(np.float32)
    b = rng.normal(0, 1, n).astype(np.float32)
    mu = rng.normal(0, 3, n).astype(np.float32)
    var = np.concatenate([rng.uniform(0, 5, n - 3), [0.0, 1e-30, 1e6]]).astype(np.float32)
    d = [torch.from_numpy(t).cuda() for t in (g, b, mu, var)]
    a1 = torch.empty(n, dtype=torch.float32, device="cuda")
    a2 = torch.empty(n, dtype=torch.float32, device="cuda")
    F.fxpq_bn_to_scale(*d, NET.BN_EPS, a1, a2)
    w1, w2 = bn_to_scale(g, b, mu, var, NET.BN_EPS)
    assert np.array_equal(a1.cpu().numpy().view(np.uint32), w1.view(np.uint32))
    assert np.array_equal(a2.cpu().numpy().view(np.uint32), w2.view(np.uint32))


@pytest.mark.parametrize("plan_seed", [7, 38])
def test_vgg16_batch64_plans(NET, plan_seed):
    _workload(NET, "vgg16", 64, 7, plan_seed=plan_seed, sample=(0,))


def test_vgg16_batch64_packed_fc_weights(NET):
    """VGG-16 with fc6 / fc7 reading packed weights (4..8 bits per the plan; fc8's are 16-bit and stay
    fp16 code planes)."""
    _workload(NET, "vgg16", 64, 7, plan_seed=7, sample=(0,), pack=True)


def test_single_conv_workload_end_to_end(NET):
    """The single-conv workload (batch 8, 64 -> 64 channels, 32 x 32 maps, 3 x 3, stride 1, pad 1): He-normal
    weights, ReLU(N(0,1)) inputs, N(0, 0.01) biases, 8-bit weights and activations with FL searched over
    0..15 (16-bit bias), the output requantized to 8 bits with its FL searched on the exact C-Block output.
    Every format and every code equals the oracle's."""
    import oracle
    from paper_2203_12091_gb300 import fxpq as F
    N, H, C, K = 8, 32, 64, 64
    g = torch.Generator().manual_seed(91)
    x = torch.relu(torch.randn(N, H, H, C, generator=g)).numpy()
    w = (torch.randn(K, 3, 3, C, generator=g) * np.sqrt(2.0 / (9 * C))).numpy().astype(np.float32)
    b = (torch.randn(K, generator=g) * 0.01).numpy().astype(np.float32)
    fmt_gpu, fmt_ora = {}, {}
    for nm, t, k in (("x", x, 8), ("w", w, 8), ("b", b, 16)):
        err, best, st = F.fl_search(torch.from_numpy(t).cuda().reshape(-1), -1, k, k, 0, 15)
        S = F.stats_from_device(st).is_signed
        fmt_gpu[nm] = F.fmt(k, S, int(best.cpu()[0]))
        _, obest, oS, _ = oracle.fl_search(t.reshape(-1), -1, k, k, 0, 15)
        fmt_ora[nm] = (k, oS, int(obest[0]))
        assert fmt_gpu[nm].tup() == fmt_ora[nm], nm
    xq = torch.empty(N * H * H * C, dtype=torch.float16, device="cuda")
    F.fxpq_quantize_rows(torch.from_numpy(x).cuda(), N * H * H, C, fmt_gpu["x"], C, xq)
    wq = torch.empty(K * 9 * C, dtype=torch.float16, device="cuda")
    F.fxpq_quantize_rows(torch.from_numpy(w).cuda(), K * 9, C, fmt_gpu["w"], C, wq)
    bq = torch.empty(K, dtype=torch.int32, device="cuda")
    F.fxpq_quantize(torch.from_numpy(b).cuda(), fmt_gpu["b"], F.DT_I32, bq)
    # the exact C-Block output's fp32 image, its FL search, then the codes
    f32 = torch.empty(N * H * H * K, dtype=torch.float32, device="cuda")
    d = F.conv_desc(N, H, H, C, C, K, 3, 3, 1, 1, True, F.OUT_F32, fmt_gpu["x"], fmt_gpu["w"], fmt_gpu["b"], None)
    F.fxpq_conv_fwd(d, xq, wq, bq, f32)
    _, ybest, yst = F.fl_search(f32, -1, 8, 8, 0, 15)
    fy = F.fmt(8, F.stats_from_device(yst).is_signed, int(ybest.cpu()[0]))
    y = torch.empty(N * H * H * K, dtype=torch.float16, device="cuda")
    d = F.conv_desc(N, H, H, C, C, K, 3, 3, 1, 1, True, F.OUT_CODES, fmt_gpu["x"], fmt_gpu["w"], fmt_gpu["b"], fy)
    F.fxpq_conv_fwd(d, xq, wq, bq, y)
    torch.cuda.synchronize()
    qx = oracle.quantize(x, *fmt_ora["x"]).reshape(x.shape)
    qw = oracle.quantize(w, *fmt_ora["w"]).reshape(w.shape)
    qb = oracle.quantize(b, *fmt_ora["b"])
    v, s = oracle.cblock(oracle.conv2d(qx, qw, 1, 1), fmt_ora["x"][2] + fmt_ora["w"][2], qb, fmt_ora["b"][2], True)
    assert np.array_equal(f32.cpu().numpy().reshape(v.shape), oracle.to_f32(v, s))
    _, oyb, oyS, _ = oracle.fl_search(oracle.to_f32(v, s).reshape(-1), -1, 8, 8, 0, 15)
    assert fy.tup() == (8, oyS, int(oyb[0]))
    want = oracle.requant(v, s, 8, oyS, int(oyb[0]))
    assert np.array_equal(F.codes_to_int(y.cpu(), fy, (N, H, H, K)).numpy(), want)
