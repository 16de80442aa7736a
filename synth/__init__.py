"""Seeded synthetic inputs shared by the CUDA path's tests/bench and the oracle.

This module holds no arithmetic of the quantization method: only random number
generation (torch.Generator on the CPU, so both sides see the same fp32 bytes),
the layer lists of the three architectures the paper evaluates (Sec. V-A), and
the seeded per-layer wordlength plans of the five workloads.  ImageNet and the
Caffe-zoo weights are not available, so images are per-channel N(0,1) (the
distribution after mean/std normalisation), weights are He-normal
(std sqrt(2 / fan_in)) and biases N(0, 0.01).
"""
from __future__ import annotations

import numpy as np
import torch


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return g


def normal(n: int, seed: int, std: float = 1.0) -> np.ndarray:
    return (torch.randn(int(n), generator=_gen(seed), dtype=torch.float32) * std).numpy()


def laplace(n: int, seed: int, scale: float = 0.1) -> np.ndarray:
    # inverse CDF of Laplace(0, scale) from U(-1/2, 1/2)
    u = torch.rand(int(n), generator=_gen(seed), dtype=torch.float64) - 0.5
    u = u.clamp(-0.5 + 1e-12, 0.5 - 1e-12)
    x = -scale * torch.sign(u) * torch.log1p(-2.0 * u.abs())
    return x.to(torch.float32).numpy()


def relu_normal(n: int, seed: int) -> np.ndarray:
    return np.maximum(normal(n, seed), np.float32(0.0))


SWEEP_DISTS = {"normal": normal, "laplace": laplace, "relu_normal": relu_normal}


def sweep_tensor(dist: str, n: int, seed: int) -> np.ndarray:
    """Standalone fp32 tensors of the FL-search sweep: N(0,1), Laplace(0, 0.1), ReLU(N(0,1))."""
    return SWEEP_DISTS[dist](n, seed)


def images(batch: int, seed: int, hw: int = 224, c: int = 3) -> np.ndarray:
    """fp32 NCHW images, per-channel N(0,1) (ImageNet statistics after normalisation)."""
    return torch.randn(batch, c, hw, hw, generator=_gen(seed), dtype=torch.float32).numpy()


# --------------------------------------------------------------------------
# Architectures (Sec. V-A).  Conv weights are KRSC (out, kh, kw, in); an FC layer is a
# convolution whose window covers the whole input map (flatten order H, W, C).
# --------------------------------------------------------------------------
def _conv(name, cin, cout, r, stride, pad, relu=True, src=None):
    return {"type": "conv", "name": name, "C": cin, "K": cout, "R": r, "stride": stride, "pad": pad,
            "relu": relu, "src": src}


def alexnet():
    """AlexNet, five CONV + three FC, groups = 1, conv1 padding 2 (55x55 map), ReLU after every
    layer but the last, MAX-POOL 3/2 after conv1, conv2 and conv5.  BN is absent (folded)."""
    L = [
        _conv("conv1", 3, 96, 11, 4, 2), {"type": "maxpool", "name": "pool1", "k": 3, "stride": 2, "pad": 0},
        _conv("conv2", 96, 256, 5, 1, 2), {"type": "maxpool", "name": "pool2", "k": 3, "stride": 2, "pad": 0},
        _conv("conv3", 256, 384, 3, 1, 1), _conv("conv4", 384, 384, 3, 1, 1), _conv("conv5", 384, 256, 3, 1, 1),
        {"type": "maxpool", "name": "pool5", "k": 3, "stride": 2, "pad": 0},
        _conv("fc6", 256, 4096, 6, 1, 0), _conv("fc7", 4096, 4096, 1, 1, 0), _conv("fc8", 4096, 1000, 1, 1, 0, relu=False),
    ]
    return L


def vgg16():
    """VGG-16, configuration D: 13 CONV 3x3/1 pad 1 in five groups, each group followed by MAX-POOL 2/2,
    then FC 25088-4096-4096-1000."""
    L = []
    cin = 3
    for g, (n, c) in enumerate([(2, 64), (2, 128), (3, 256), (3, 512), (3, 512)], start=1):
        for i in range(1, n + 1):
            L.append(_conv(f"conv{g}_{i}", cin, c, 3, 1, 1))
            cin = c
        L.append({"type": "maxpool", "name": f"pool{g}", "k": 2, "stride": 2, "pad": 0})
    L += [_conv("fc6", 512, 4096, 7, 1, 0), _conv("fc7", 4096, 4096, 1, 1, 0), _conv("fc8", 4096, 1000, 1, 1, 0, relu=False)]
    return L


def resnet18(bn: bool = False):
    """ResNet-18 (torchvision topology), BN folded into each conv as a bias, or (bn=True) kept as a
    Scale layer after a bias-free conv (the Caffe ResNet form: CONV, BatchNorm, Scale, ReLU).  Stage 1
    uses identity shortcuts; stages 2-4 open with a 1x1/2 downsample shortcut.  Every conv output,
    and every residual add (+ReLU), is a C-Block followed by a QLayer; MAX-POOL has none; the global
    AVG-POOL multiplies by the quantized reciprocal 1/49."""
    L = [_conv("conv1", 3, 64, 7, 2, 3), {"type": "maxpool", "name": "pool1", "k": 3, "stride": 2, "pad": 1}]
    cin = 64
    prev = "pool1"
    for stage, c in enumerate([64, 128, 256, 512], start=1):
        for blk in range(2):
            stride = 2 if (stage > 1 and blk == 0) else 1
            pfx = f"res{stage}{'ab'[blk]}"
            L.append(_conv(pfx + "_branch2a", cin, c, 3, stride, 1, relu=True, src=prev))
            L.append(_conv(pfx + "_branch2b", c, c, 3, 1, 1, relu=False, src=pfx + "_branch2a"))
            if stride != 1 or cin != c:
                L.append(_conv(pfx + "_branch1", cin, c, 1, stride, 0, relu=False, src=prev))
                short = pfx + "_branch1"
            else:
                short = prev
            L.append({"type": "eltwise", "name": pfx, "a": pfx + "_branch2b", "b": short, "relu": True})
            prev = pfx
            cin = c
    if bn:
        for layer in L:
            if layer["type"] == "conv":
                layer["bn"] = True
    L.append({"type": "avgpool", "name": "pool5", "src": prev})
    L.append(_conv("fc", 512, 1000, 1, 1, 0, relu=False, src="pool5"))
    return L


def resnet18_bn():
    return resnet18(bn=True)


ARCHS = {"alexnet": alexnet, "vgg16": vgg16, "resnet18": resnet18, "resnet18_bn": resnet18_bn}


def weights(arch: str, seed: int):
    """He-normal fp32 weights (std sqrt(2 / (C*R*R))) in KRSC and N(0, 0.01) biases, per conv/FC layer;
    a conv followed by a BN layer has no bias (None)."""
    g = _gen(seed)
    out = {}
    for L in ARCHS[arch]():
        if L["type"] != "conv":
            continue
        fan_in = L["C"] * L["R"] * L["R"]
        w = torch.randn(L["K"], L["R"], L["R"], L["C"], generator=g, dtype=torch.float32) * float(np.sqrt(2.0 / fan_in))
        if L.get("bn"):
            out[L["name"]] = (w.numpy(), None)
            continue
        b = torch.randn(L["K"], generator=g, dtype=torch.float32) * 0.01
        out[L["name"]] = (w.numpy(), b.numpy())
    return out


def bn_params(arch: str, seed: int):
    """Per BN layer (a conv with "bn"): fp32 (gamma, beta, running mean, running variance) of its K
    channels, drawn as gamma ~ U(0.5, 1.5), beta ~ N(0, 0.2), mean ~ N(0, 0.2), var ~ U(0.5, 2.0)
    (no trained statistics exist; these keep the per-channel gain aleph1 within about [0.35, 2.1])."""
    g = _gen(seed)
    out = {}
    for L in ARCHS[arch]():
        if L["type"] != "conv" or not L.get("bn"):
            continue
        K = L["K"]
        gamma = torch.rand(K, generator=g, dtype=torch.float32) + 0.5
        beta = torch.randn(K, generator=g, dtype=torch.float32) * 0.2
        mean = torch.randn(K, generator=g, dtype=torch.float32) * 0.2
        var = torch.rand(K, generator=g, dtype=torch.float32) * 1.5 + 0.5
        out[L["name"]] = tuple(t.numpy() for t in (gamma, beta, mean, var))
    return out


def bit_plan(arch: str, seed: int):
    """Per-layer wordlengths of the workloads.

    alexnet : 8-bit weights and activations (input included), 16-bit biases.
    resnet18: weight bits drawn from {3..8}, activation bits from {4..8} (seeded), 16-bit biases,
              16-bit unsigned AVG-POOL reciprocal.
    resnet18_bn: resnet18's draws; each BN layer's Scale parameters aleph1 ("s") and aleph2 ("h")
              16-bit (the C-Block's 16-bit multiplier, Sec. IV-B) in place of the bias.
    vgg16   : first and last layers 16-bit (input image, conv1_1 weights, fc7 output and fc8 weights),
              every other weight / activation drawn from {4..8} (seeded), 16-bit biases.
    Returns {"input": a_bits, layer_name: {"w": .., "b": .., "a": ..}} where "a" is the wordlength of
    the layer's output QLayer (absent for the last layer and for MAX-POOL).
    """
    rng = np.random.default_rng(seed)
    layers = ARCHS[arch]()
    names = [L["name"] for L in layers]
    plan = {}
    if arch == "alexnet":
        plan["input"] = 8
        for L in layers:
            if L["type"] == "conv":
                plan[L["name"]] = {"w": 8, "b": 16}
                if L["name"] != "fc8":
                    plan[L["name"]]["a"] = 8
        return plan
    if arch in ("resnet18", "resnet18_bn"):
        plan["input"] = int(rng.integers(4, 9))
        for L in layers:
            if L["type"] == "conv":
                plan[L["name"]] = {"w": int(rng.integers(3, 9))}
                plan[L["name"]].update({"s": 16, "h": 16} if L.get("bn") else {"b": 16})
                if L["name"] != "fc":
                    plan[L["name"]]["a"] = int(rng.integers(4, 9))
            elif L["type"] in ("eltwise", "avgpool"):
                plan[L["name"]] = {"a": int(rng.integers(4, 9))}
                if L["type"] == "avgpool":
                    plan[L["name"]]["r"] = 16
        return plan
    if arch == "vgg16":
        convs = [L["name"] for L in layers if L["type"] == "conv"]
        plan["input"] = 16
        for nm in convs:
            plan[nm] = {"w": int(rng.integers(4, 9)), "b": 16}
            if nm != "fc8":
                plan[nm]["a"] = int(rng.integers(4, 9))
        plan["conv1_1"]["w"] = 16
        plan["fc7"]["a"] = 16
        plan["fc8"]["w"] = 16
        return plan
    raise ValueError(arch)


def macs_per_image(arch: str, hw: int = 224) -> int:
    """Multiply-accumulates per image of the conv/FC layers (pool/eltwise excluded)."""
    layers = ARCHS[arch]()
    shapes = {}
    h, c = hw, 3
    total = 0
    prev = None
    for L in layers:
        src = L.get("src") or prev
        if src is not None:
            h, c = shapes[src]
        if L["type"] == "conv":
            p = (h + 2 * L["pad"] - L["R"]) // L["stride"] + 1
            total += p * p * L["K"] * L["C"] * L["R"] * L["R"]
            shapes[L["name"]] = (p, L["K"])
        elif L["type"] == "maxpool":
            p = (h + 2 * L["pad"] - L["k"]) // L["stride"] + 1
            shapes[L["name"]] = (p, c)
        elif L["type"] == "eltwise":
            shapes[L["name"]] = shapes[L["a"]]
        elif L["type"] == "avgpool":
            shapes[L["name"]] = (1, c)
        prev = L["name"]
    return total
