"""Seeded synthetic inputs for the integer-only convolution workloads.

This module only draws random integers (codes and per-channel parameters) with numpy's
``default_rng(seed)``; it holds none of the method's arithmetic (no packing, no
convolution, no rescale). Both the CUDA path and the CPU oracle consume what it returns.

Shapes follow the detector workloads of the paper's experiments (Sec. 4: RetinaNet/FCOS
with a ResNet backbone, FPN levels P3-P7, images resized to an 800-pixel short side).
The images themselves (COCO) are not used: codes are drawn from the distributions below.

Draw order per conv: activation codes, weight codes, M0, shift, bias, then the skip
parameters (c, d) and the skip tensor.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# FPN levels P3..P7 for an 800x1333 image zero-padded to 800x1344 (a multiple of 32, so
# every 2x upsample-add lines up): strides 8..128.
FPN_LEVELS = [(100, 168), (50, 84), (25, 42), (13, 21), (7, 11)]


def act_codes(rng, shape, bits: int, dist: str = "uniform") -> np.ndarray:
    """Unsigned k-bit activation codes (Eq. 2 range [0, 2^k - 1])."""
    hi = (1 << bits) - 1
    if dist == "uniform":
        return rng.integers(0, hi + 1, size=shape, dtype=np.int32)
    if dist == "halfnormal4":  # |N(0, 4)| rounded, clipped to the code range
        v = np.abs(rng.normal(0.0, 4.0, size=shape))
        return np.clip(np.floor(v + 0.5), 0, hi).astype(np.int32)
    raise ValueError(dist)


def weight_codes(rng, shape, bits: int, dist: str = "uniform") -> np.ndarray:
    """Signed weight integers, symmetric range [-(2^(k-1)-1), 2^(k-1)-1]."""
    lim = (1 << (bits - 1)) - 1
    if dist == "uniform":
        return rng.integers(-lim, lim + 1, size=shape, dtype=np.int32)
    if dist == "normal2":  # N(0, 2) rounded, clipped to the range (std 2)
        v = rng.normal(0.0, 2.0, size=shape)
        return np.clip(np.floor(v + 0.5), -lim, lim).astype(np.int32)
    raise ValueError(dist)


def requant_params(rng, levels: int, cout: int, *, shift_lo: int = 8, shift_hi: int = 20,
                   bias_lim: int = 4096, calib_std: float | None = None, out_bits: int = 2):
    """M0 uniform in [2^30, 2^31), shift uniform in [shift_lo, shift_hi], bias uniform in
    [-bias_lim, bias_lim]. With ``calib_std`` (the accumulator's standard deviation), the
    shift is instead drawn around the value that spreads outputs over the k-bit range and
    the bias is drawn within one standard deviation, so outputs neither all clip nor all
    round to zero."""
    m0 = rng.integers(1 << 30, 1 << 31, size=(levels, cout), dtype=np.int64).astype(np.int32)
    if calib_std is None:
        shift = rng.integers(shift_lo, shift_hi + 1, size=(levels, cout)).astype(np.int8)
        bias = rng.integers(-bias_lim, bias_lim + 1, size=(levels, cout), dtype=np.int64).astype(np.int32)
    else:
        centre = math.log2(max(2.0 * calib_std / ((1 << out_bits) - 1), 1e-9)) - 0.5
        base = int(round(centre))
        shift = (base + rng.integers(-1, 2, size=(levels, cout))).clip(-31, 31).astype(np.int8)
        lim = max(1, int(calib_std))
        bias = rng.integers(-lim, lim + 1, size=(levels, cout), dtype=np.int64).astype(np.int32)
    return m0, shift, bias


def skip_params(rng, levels: int, cout: int, shift_main: np.ndarray):
    """Skip rescale c/2^d (Eq. 8) with c uniform in [2^30, 2^31) and d = 30 - shift + delta,
    delta uniform in {0, 1, 2}: one skip code then moves the output by 1/8 to 2 LSB."""
    c = rng.integers(1 << 30, 1 << 31, size=(levels, cout), dtype=np.int64).astype(np.int32)
    delta = rng.integers(0, 3, size=(levels, cout))
    d = np.clip(30 - shift_main.astype(np.int64) + delta, 0, 62).astype(np.int8)
    return c, d


@dataclass
class ConvSpec:
    cin: int
    cout: int
    kh: int
    kw: int
    stride: int
    pad: int
    w: np.ndarray           # [cout, kh, kw, cin] signed integers
    w_bits: int
    m0: np.ndarray | None   # [levels, cout]
    shift: np.ndarray | None
    bias: np.ndarray | None
    out_bits: int
    skip_c: np.ndarray | None = None
    skip_d: np.ndarray | None = None


@dataclass
class Workload:
    name: str
    bits: int
    inputs: list            # list of activation code arrays [n, h, w, c]
    convs: list             # list of ConvSpec
    extra: dict = field(default_factory=dict)


def config0(seed: int = 0) -> Workload:
    """Single 3x3 conv, stride 1, pad 1, batch 1, 64->64, 32x32, 2-bit."""
    rng = np.random.default_rng(seed)
    x = act_codes(rng, (1, 32, 32, 64), 2)
    w = weight_codes(rng, (64, 3, 3, 64), 2)
    m0, shift, bias = requant_params(rng, 1, 64)
    conv = ConvSpec(64, 64, 3, 3, 1, 1, w, 2, m0, shift, bias, 2)
    return Workload("conv3x3_64to64_32x32_b1_2bit", 2, [x], [conv])


def config1(seed: int = 1, batch: int = 2, h: int = 100, w: int = 152) -> Workload:
    """ResNet-50 stage-C3 bottleneck: 1x1 512->128, 3x3 128->128, 1x1 128->512 with the
    identity skip, 4-bit; activations |N(0,4)|, weights N(0,2)."""
    rng = np.random.default_rng(seed)
    x = act_codes(rng, (batch, h, w, 512), 4, "halfnormal4")
    convs = []
    for cin, cout, k, pad in ((512, 128, 1, 0), (128, 128, 3, 1), (128, 512, 1, 0)):
        wt = weight_codes(rng, (cout, k, k, cin), 4, "normal2")
        m0, shift, bias = requant_params(rng, 1, cout)
        convs.append(ConvSpec(cin, cout, k, k, 1, pad, wt, 4, m0, shift, bias, 4))
    c, d = skip_params(rng, 1, 512, convs[2].shift)
    convs[2].skip_c, convs[2].skip_d = c, d
    return Workload(f"r50_c3_bottleneck_b{batch}_{h}x{w}_4bit", 4, [x], convs)


def head_tower(seed: int, batch: int, bits: int, levels=None, name: str | None = None,
               calibrated: bool = False) -> Workload:
    """Shared detector head: 4 x [3x3 256->256, requant, ReLU-clip] over the FPN levels
    with one (M0, shift, bias) set per level (multi-level BN, Sec. 3.2.2), then a 3x3
    256->80 classification conv and a 3x3 256->4 box conv with int32 outputs."""
    levels = FPN_LEVELS if levels is None else levels
    rng = np.random.default_rng(seed)
    nl = len(levels)
    inputs = [act_codes(rng, (batch, hh, ww, 256), bits) for (hh, ww) in levels]
    convs = []
    lim = (1 << (bits - 1)) - 1
    hi = (1 << bits) - 1
    # accumulator std for uniform codes: sqrt(K * E[x^2] * E[w^2])
    ex2 = sum(v * v for v in range(hi + 1)) / (hi + 1)
    ew2 = sum(v * v for v in range(-lim, lim + 1)) / (2 * lim + 1)
    std = math.sqrt(9 * 256 * ex2 * ew2)
    for _ in range(4):
        wt = weight_codes(rng, (256, 3, 3, 256), bits)
        m0, shift, bias = requant_params(rng, nl, 256, calib_std=std if calibrated else None,
                                         out_bits=bits)
        convs.append(ConvSpec(256, 256, 3, 3, 1, 1, wt, bits, m0, shift, bias, bits))
    for cout in (80, 4):
        wt = weight_codes(rng, (cout, 3, 3, 256), bits)
        bias = rng.integers(-4096, 4097, size=(nl, cout), dtype=np.int64).astype(np.int32)
        convs.append(ConvSpec(256, cout, 3, 3, 1, 1, wt, bits, None, None, bias, 32))
    nm = name or f"head_tower_b{batch}_{bits}bit_{nl}lvl"
    return Workload(nm, bits, inputs, convs, {"levels": list(levels), "batch": batch})


def config2(seed: int = 2, calibrated: bool = False) -> Workload:
    return head_tower(seed, 2, 2, name="retina_head_800x1333_b2_2bit", calibrated=calibrated)


def config4(bits: int, seed: int = 4) -> Workload:
    return head_tower(seed, 16, bits, name=f"retina_head_800x1333_b16_{bits}bit")


def sample_pixels(rng, total: int, n: int) -> np.ndarray:
    """Distinct flattened output-pixel indices, always including the first and last."""
    n = min(n, total)
    idx = rng.choice(total, size=n, replace=False).astype(np.int64)
    idx[0] = 0
    if n > 1:
        idx[1] = total - 1
    return np.unique(idx)


# ------------------------------------------------------------------ config 3: whole network

# second moments of the drawn distributions, for the calibrated shifts below
_EX2_CODE4 = 16.0                     # |N(0,4)| clipped to [0, 15]: E[x^2] ~ 16
_EX2_CODE8 = sum(v * v for v in range(256)) / 256.0   # uniform 8-bit image codes
_EW2_NORMAL2 = 4.0                    # N(0, 2) clipped to [-7, 7]: E[w^2] ~ 4


def skip_params_acc(rng, levels: int, cout: int):
    """Rescale c/2^d of an int32 skip held in another conv's accumulator units (a downsample
    branch): c uniform in [2^30, 2^31), d = 31 + delta with delta uniform in {0, 1, 2}, so the
    branch enters the sum at 1/8 to 1 times its own value."""
    c = rng.integers(1 << 30, 1 << 31, size=(levels, cout), dtype=np.int64).astype(np.int32)
    d = (31 + rng.integers(0, 3, size=(levels, cout))).astype(np.int8)
    return c, d


@dataclass
class Layer:
    """One step of a network: a conv (``conv`` set) or a max-pool on codes (``pool`` set).
    ``src``, ``dst`` and ``skip`` name tensors, one entry per job; a grouped layer (the shared
    head) has one job per FPN level, and job l uses row l of the per-level tables. ``upsample``
    2 reads the skip at half resolution (nearest 2x, the FPN top-down add)."""
    name: str
    src: list
    dst: list
    conv: ConvSpec | None = None
    skip: list | None = None
    upsample: int = 1
    pool: tuple | None = None     # (k, stride, pad)


def _conv(rng, cin, cout, k, stride, pad, *, levels=1, out_bits=4, x_ex2=_EX2_CODE4, w_bits=4,
          skip="none", skip_levels=None):
    """Draws one conv in the fixed order: weights, M0, shift, bias, then the skip's (c, d).
    Codes out: requant calibrated from the accumulator's standard deviation. int32 out: bias only."""
    wt = weight_codes(rng, (cout, k, k, cin), 4, "normal2")
    std = math.sqrt(k * k * cin * x_ex2 * _EW2_NORMAL2)
    if out_bits == 32:
        lim = max(1, int(std))
        bias = rng.integers(-lim, lim + 1, size=(levels, cout), dtype=np.int64).astype(np.int32)
        cv = ConvSpec(cin, cout, k, k, stride, pad, wt, w_bits, None, None, bias, 32)
    else:
        m0, shift, bias = requant_params(rng, levels, cout, calib_std=std, out_bits=out_bits)
        cv = ConvSpec(cin, cout, k, k, stride, pad, wt, w_bits, m0, shift, bias, out_bits)
    if skip == "codes":
        cv.skip_c, cv.skip_d = skip_params(rng, levels, cout, cv.shift)
    elif skip == "acc":
        cv.skip_c, cv.skip_d = skip_params_acc(rng, levels, cout)
    return cv


def config3(seed: int = 3, batch: int = 8, h: int = 800, w: int = 1333, w_pad: int = 1344) -> Workload:
    """Integer ResNet-18 backbone + FPN (P3-P7, 256 channels) + the shared head of config 2,
    4-bit weights (N(0,2) rounded, clipped to [-7, 7]) and 4-bit activations; the input is an
    8-bit RGB image batch (codes uniform in [0, 255]) zero-padded on the right from w to w_pad
    columns. Every conv's requant is calibrated so that activations stay spread over the code
    range through the depth of the network.

    Layers (NHWC, codes unless stated):
    - conv1 7x7 s2 p3 3->64 (8-bit input; weights held as 8-bit codes since a 3-channel row has
      no 4-bit packed layout), max-pool 3x3 s2 p1;
    - four stages of two basic blocks (64, 128, 256, 512 channels; stages 2-4 start with a 3x3 s2
      conv and a 1x1 s2 downsample conv whose int32 output is the block's skip, Eq. 7 with
      an accumulator-domain operand); identity skips are the block input's codes;
    - FPN: 1x1 lateral convs on C3, C4, C5; the top-down path adds the coarser merged map,
      read with nearest 2x upsampling, in the lateral conv's epilogue (Eq. 7); 3x3 output convs
      give P3-P5; P6 = 3x3 s2 on C5, P7 = 3x3 s2 on P6;
    - head: 4 x [3x3 256->256] over P3-P7 with per-level (M0, shift, bias) (Sec. 3.2.2), then
      3x3 256->80 classification and 3x3 256->4 box convs with int32 outputs.
    """
    rng = np.random.default_rng(seed)
    x = np.zeros((batch, h, w_pad, 3), dtype=np.int32)
    x[:, :, :w] = act_codes(rng, (batch, h, w, 3), 8)
    layers: list[Layer] = []
    c1 = _conv(rng, 3, 64, 7, 2, 3, x_ex2=_EX2_CODE8, w_bits=8)
    layers.append(Layer("conv1", ["image"], ["conv1"], conv=c1))
    layers.append(Layer("pool", ["conv1"], ["pool"], pool=(3, 2, 1)))
    cur, cin = "pool", 64
    for stage, cout in enumerate((64, 128, 256, 512), start=1):
        for blk in range(2):
            down = stage > 1 and blk == 0
            pre = f"layer{stage}.{blk}"
            a = _conv(rng, cin, cout, 3, 2 if down else 1, 1)
            layers.append(Layer(pre + ".conv_a", [cur], [pre + ".a"], conv=a))
            if down:
                ds = _conv(rng, cin, cout, 1, 2, 0, out_bits=32)
                layers.append(Layer(pre + ".down", [cur], [pre + ".down"], conv=ds))
                b = _conv(rng, cout, cout, 3, 1, 1, skip="acc")
                layers.append(Layer(pre + ".conv_b", [pre + ".a"], [pre], conv=b, skip=[pre + ".down"]))
            else:
                b = _conv(rng, cout, cout, 3, 1, 1, skip="codes")
                layers.append(Layer(pre + ".conv_b", [pre + ".a"], [pre], conv=b, skip=[cur]))
            cur, cin = pre, cout
    c3, c4, c5 = "layer2.1", "layer3.1", "layer4.1"
    layers.append(Layer("fpn.lat5", [c5], ["fpn.m5"], conv=_conv(rng, 512, 256, 1, 1, 0)))
    layers.append(Layer("fpn.lat4", [c4], ["fpn.m4"], conv=_conv(rng, 256, 256, 1, 1, 0, skip="codes"),
                        skip=["fpn.m5"], upsample=2))
    layers.append(Layer("fpn.lat3", [c3], ["fpn.m3"], conv=_conv(rng, 128, 256, 1, 1, 0, skip="codes"),
                        skip=["fpn.m4"], upsample=2))
    for l in (3, 4, 5):
        layers.append(Layer(f"fpn.out{l}", [f"fpn.m{l}"], [f"P{l}"], conv=_conv(rng, 256, 256, 3, 1, 1)))
    layers.append(Layer("fpn.p6", [c5], ["P6"], conv=_conv(rng, 512, 256, 3, 2, 1)))
    layers.append(Layer("fpn.p7", ["P6"], ["P7"], conv=_conv(rng, 256, 256, 3, 2, 1)))
    src = [f"P{l}" for l in range(3, 8)]
    for i in range(4):
        dst = [f"head.t{i}.{l}" for l in range(5)]
        layers.append(Layer(f"head.tower{i}", src, dst, conv=_conv(rng, 256, 256, 3, 1, 1, levels=5)))
        src = dst
    layers.append(Layer("head.cls", src, [f"cls.{l}" for l in range(5)],
                        conv=_conv(rng, 256, 80, 3, 1, 1, levels=5, out_bits=32)))
    layers.append(Layer("head.box", src, [f"box.{l}" for l in range(5)],
                        conv=_conv(rng, 256, 4, 3, 1, 1, levels=5, out_bits=32)))
    name = f"int_resnet18_fpn_retina_b{batch}_{h}x{w_pad}_4bit"
    return Workload(name, 4, [x], [ly.conv for ly in layers if ly.conv is not None],
                    {"layers": layers, "batch": batch, "hw": (h, w_pad), "input_bits": 8})
