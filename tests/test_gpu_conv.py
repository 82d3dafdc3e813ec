"""GPU parity of the integer convolution (Eq. 4 + fused Eq. 6/7/2 epilogue) against the
CPU oracle: bit-exact on every output byte, through the C ABI, for both kernels."""
import numpy as np
import pytest

from gpu_util import assert_same, conv_pair, weights
from paper_2007_06919_gb300 import synth

pytestmark = pytest.mark.gpu

TC, DIRECT, TC_NO_PAIR, TC_NO_FP4, TC_NO_PAIR_NO_FP4 = 1, 2, 3, 4, 5
FP4 = 6  # reported path of the FP4 tensor-core pipe


def ws_path(cout: int) -> int:
    """Path reported for the workspace-fed tensor-core kernel: it runs on CTA pairs (4)."""
    return 4


def fp4_applies(xb, wb, fmt, cin, cout):
    """Whether a workspace-path conv runs on the FP4 pipe: 2-bit codes, weights exact as E2M1
    w / 2 (|w| <= 4), cin % 256 == 0, at most 240 channels per N tile."""
    max_w = (1 << (wb - 1)) if fmt == 0 else (1 << wb) - 1
    bn = (cout + 15) // 16 * 16 if cout <= 256 else 256
    return xb == 2 and max_w <= 4 and cin % 256 == 0 and bn <= 240


def _params(rng, levels, cout, out_bits, calib_std=None):
    return synth.requant_params(rng, levels, cout, calib_std=calib_std, out_bits=out_bits)


def test_library_uses_the_gpu():
    import torch
    assert torch.cuda.is_available()
    cap = torch.cuda.get_device_capability()
    assert cap[0] >= 10, cap


@pytest.mark.parametrize("path", [TC, DIRECT])
def test_config0_bit_exact(path):
    wl = synth.config0()
    cv = wl.convs[0]
    got, want, used = conv_pair(wl.inputs[0], 2, cv.w, 2, m0=cv.m0, shift=cv.shift, bias=cv.bias,
                                out_bits=2, path=path)
    assert used == path
    assert_same(got, want, 64, 2, "config0")


@pytest.mark.parametrize("path", [TC, DIRECT])
def test_config0_calibrated_bit_exact(path):
    """Same shape with shifts drawn so codes spread over 0..3 (not all clipped)."""
    rng = np.random.default_rng(100)
    x = synth.act_codes(rng, (1, 32, 32, 64), 2)
    w = synth.weight_codes(rng, (64, 3, 3, 64), 2)
    m0, sh, b = _params(rng, 1, 64, 2, calib_std=37.0)
    got, want, _ = conv_pair(x, 2, w, 2, m0=m0, shift=sh, bias=b, out_bits=2, path=path)
    assert len(np.unique(got)) > 8
    assert_same(got, want, 64, 2, "config0 calibrated")


# (x_bits, w_bits, w_format, n, h, w, cin, cout, k, stride, pad, out_bits)
CASES = [
    (2, 2, 0, 2, 13, 17, 64, 64, 3, 1, 1, 2),      # ragged M (442 rows), K = 576
    (4, 4, 0, 1, 9, 23, 128, 128, 3, 1, 1, 4),     # 4-bit, ragged
    (3, 3, 0, 2, 7, 11, 96, 64, 3, 1, 1, 3),       # 3-bit, cin 96: a 128-byte chunk spans taps
    (2, 2, 1, 1, 10, 10, 32, 32, 3, 1, 1, 2),      # Eq. 3 odd weights, cin 32 (K = 288 -> 384)
    (4, 4, 1, 1, 6, 9, 64, 64, 3, 1, 1, 4),        # odd 4-bit weights: |w| up to 15
    (4, 4, 0, 2, 15, 14, 64, 128, 3, 2, 1, 4),     # stride 2
    (4, 4, 0, 2, 16, 12, 512, 128, 1, 1, 0, 4),    # 1x1 512 -> 128
    (4, 4, 0, 1, 8, 8, 128, 512, 1, 1, 0, 4),      # 1x1 128 -> 512: two N tiles
    (4, 2, 0, 1, 19, 21, 32, 64, 7, 2, 3, 4),      # 7x7 stride 2
    (2, 2, 0, 2, 11, 9, 256, 80, 3, 1, 1, 32),     # int32 output, 80 channels (N tile 80)
    (2, 2, 0, 2, 5, 7, 256, 4, 3, 1, 1, 32),       # int32 output, 4 channels (N tile 16)
    (2, 2, 0, 1, 1, 1, 64, 64, 3, 1, 1, 2),        # 1x1 image: every tap but the centre pads
    (4, 4, 0, 1, 3, 300, 64, 32, 1, 1, 0, 8),      # 8-bit output codes
    (3, 4, 0, 1, 33, 5, 32, 96, 3, 1, 0, 3),       # no padding, cout 96
    (4, 4, 0, 2, 9, 13, 192, 64, 3, 1, 1, 4),      # cin 192: three 64-channel chunks per tap
]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
@pytest.mark.parametrize("path", [TC, DIRECT])
def test_conv_shapes_bit_exact(case, path):
    xb, wb, fmt, n, h, wd, cin, cout, k, stride, pad, ob = case
    rng = np.random.default_rng(hash(case) % 2 ** 32)
    x = synth.act_codes(rng, (n, h, wd, cin), xb)
    if fmt == 0:
        w = rng.integers(-(1 << (wb - 1)), 1 << (wb - 1), size=(cout, k, k, cin)).astype(np.int32)
    else:
        w = rng.integers(0, 1 << wb, size=(cout, k, k, cin)).astype(np.int32)
    std = np.sqrt(k * k * cin * np.mean(np.arange(1 << xb) ** 2) * (1 << (2 * wb - 2)) / 3)
    m0, sh, b = _params(rng, 1, cout, ob if ob != 32 else 4, calib_std=std)
    got, want, used = conv_pair(x, xb, w, wb, w_format=fmt, stride=stride, pad=pad, out_bits=ob,
                                m0=m0, shift=sh, bias=b, path=path)
    assert used == path
    assert_same(got, want, cout, ob, f"case {case}")


# workspace path: 128-byte K chunks (cin % 128 == 0) or 64-byte ones (cin % 64 == 0)
WS_CASES = [c for c in CASES if c[9] == 1 and c[6] % 64 == 0 and c[0] <= 4 and c[1] <= 4]


@pytest.mark.parametrize("case", WS_CASES, ids=[str(i) for i in range(len(WS_CASES))])
@pytest.mark.parametrize("pairs", [True, False])
@pytest.mark.parametrize("fp4", [True, False])
def test_conv_workspace_path_bit_exact(case, pairs, fp4):
    """The expanded-activation path (one expansion pass into a caller workspace, then TMA
    tiles of the zero-padded byte or nibble image, junk columns dropped) gives the same
    bytes, on CTA pairs (256-wide N tiles) and on single CTAs, on the E4M3 pipe and, where
    it applies, on the FP4 one."""
    xb, wb, fmt, n, h, wd, cin, cout, k, stride, pad, ob = case
    rng = np.random.default_rng(hash(case) % 2 ** 32 + 1)
    x = synth.act_codes(rng, (n, h, wd, cin), xb)
    w = rng.integers(-(1 << (wb - 1)), 1 << (wb - 1), size=(cout, k, k, cin)).astype(np.int32)
    std = np.sqrt(k * k * cin * np.mean(np.arange(1 << xb) ** 2) * (1 << (2 * wb - 2)) / 3)
    m0, sh, b = _params(rng, 1, cout, ob if ob != 32 else 4, calib_std=std)
    mode = {(True, True): TC, (True, False): TC_NO_FP4, (False, True): TC_NO_PAIR,
            (False, False): TC_NO_PAIR_NO_FP4}[(pairs, fp4)]
    got, want, used = conv_pair(x, xb, w, wb, stride=stride, pad=pad, out_bits=ob, m0=m0, shift=sh, bias=b,
                                path=mode, workspace=True)
    assert used == (FP4 if fp4 and fp4_applies(xb, wb, fmt, cin, cout) else (ws_path(cout) if pairs else 3))
    assert_same(got, want, cout, ob, f"workspace case {case}")


@pytest.mark.parametrize("shape", [(1, 1, 1), (2, 3, 300), (1, 37, 2), (3, 7, 11)])
@pytest.mark.parametrize("pairs", [True, False])
def test_workspace_path_edge_shapes(shape, pairs):
    """Tiles that cross image rows and images, 1x1 images and single-column images."""
    n, h, wd = shape
    rng = np.random.default_rng(n * 1000 + h * 10 + wd)
    x = synth.act_codes(rng, (n, h, wd, 256), 2)
    w = synth.weight_codes(rng, (256, 3, 3, 256), 2)
    m0, sh, b = _params(rng, 1, 256, 2, calib_std=37.0)
    got, want, used = conv_pair(x, 2, w, 2, out_bits=2, m0=m0, shift=sh, bias=b,
                                path=TC if pairs else TC_NO_PAIR, workspace=True)
    assert used == (4 if pairs else 3)
    assert_same(got, want, 256, 2, f"edge {shape}")


@pytest.mark.parametrize("path", [TC, DIRECT])
@pytest.mark.parametrize("skip_bits,upsample,mirror", [(4, 1, 0), (4, 1, 1), (32, 1, 0), (2, 2, 0), (32, 2, 1),
                                                        (8, 1, 0), (32, 2, 0)])
@pytest.mark.parametrize("ws", [False, True])
def test_conv_with_skip_bit_exact(path, skip_bits, upsample, mirror, ws):
    """Eq. 7 fused into the epilogue: identity / downsample (int32) / FPN (upsample 2) skips,
    both directions of the rescale."""
    rng = np.random.default_rng(7 + skip_bits + 10 * upsample + 100 * mirror)
    n, h, wd, cin, cout = 2, 14, 11, 128, 64
    x = synth.act_codes(rng, (n, h, wd, cin), 4)
    w = synth.weight_codes(rng, (cout, 3, 3, cin), 4, "normal2")
    m0, sh, b = _params(rng, 1, cout, 4, calib_std=300.0)
    sh_ = (h + upsample - 1) // upsample, (wd + upsample - 1) // upsample
    if skip_bits == 32:
        skip = rng.integers(-5000, 5000, size=(n, sh_[0], sh_[1], cout)).astype(np.int32)
    else:
        skip = synth.act_codes(rng, (n, sh_[0], sh_[1], cout), skip_bits)
    c, d = synth.skip_params(rng, 1, cout, sh)
    got, want, used = conv_pair(x, 4, w, 4, out_bits=4, m0=m0, shift=sh, bias=b, skip=skip, skip_bits=skip_bits,
                             skip_c=c, skip_d=d, upsample=upsample, scale_main=mirror, path=path, workspace=ws)
    assert used == (4 if (ws and path == TC) else path)
    assert_same(got, want, cout, 4, "skip")


@pytest.mark.parametrize("x_bits,w_lim", [(4, 8), (3, 4), (2, 2)])
def test_tensor_core_sum_is_exact_at_the_bound(x_bits, w_lim):
    """Adversarial accumulation: every code at its maximum and weights of one sign, with
    K as large as the exact-FP32 bound K * max|x| * max|w| < 2^24 lets the tensor-core
    kernel take; int32 outputs must equal the oracle's int64 sums exactly."""
    amax = (1 << x_bits) - 1
    cin = 32 * ((((1 << 24) - 1) // (9 * amax * w_lim)) // 32)
    cin = min(cin, 65536)
    rng = np.random.default_rng(x_bits)
    x = np.full((1, 5, 6, cin), amax, np.int32)
    x[0, 2, 3, ::3] = rng.integers(0, amax + 1, size=x[0, 2, 3, ::3].shape)
    w = np.full((32, 3, 3, cin), -w_lim, np.int32)
    w[1::2] = w_lim - 1 if w_lim - 1 > 0 else 1     # odd channels positive
    w[5, :, :, ::2] = 1                              # mixed signs inside one sum
    got, want, used = conv_pair(x, x_bits, w, 4 if w_lim == 8 else (3 if w_lim == 4 else 2), pad=1,
                                out_bits=32, bias=np.zeros((1, 32), np.int32), path=TC)
    assert used == TC
    assert_same(got, want, 32, 32, "exactness")
    assert np.abs(want.view(np.int32)).max() > (1 << 21)


def test_paths_agree_on_config1_conv2():
    """3x3 128->128 4-bit of the bottleneck at full size on both kernels and the oracle."""
    wl = synth.config1()
    cv = wl.convs[1]
    rng = np.random.default_rng(5)
    x = synth.act_codes(rng, (2, 100, 152, 128), 4, "halfnormal4")
    wp = weights(cv.w, 4)
    outs = [conv_pair(x, 4, cv.w, 4, m0=cv.m0, shift=cv.shift, bias=cv.bias, out_bits=4, path=p, wprep=wp)
            for p in (TC, DIRECT)]
    assert_same(outs[0][0], outs[0][1], 128, 4, "tc")
    assert_same(outs[1][0], outs[1][1], 128, 4, "direct")


def test_invalid_skip_shape_is_rejected_before_launch():
    import torch
    from paper_2007_06919_gb300 import aqd
    rng = np.random.default_rng(0)
    W, _ = weights(synth.weight_codes(rng, (32, 3, 3, 32), 2), 2)
    X = aqd.DTensor.empty(1, 8, 8, 32, 2)
    Y = aqd.DTensor.empty(1, 8, 8, 32, 2)
    S = aqd.DTensor.empty(1, 3, 8, 32, 2)  # too few rows for the output
    rq = aqd.RequantParams.from_numpy(np.ones((1, 32)), np.zeros((1, 32)), np.zeros((1, 32)))
    sp = aqd.SkipParams.from_numpy(np.ones((1, 32)), np.zeros((1, 32)))
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int(X, W, 1, 1, Y, rq=rq, skip=S, sp=sp)
    assert e.value.status == 1
    torch.cuda.synchronize()


STEM = 5


@pytest.mark.parametrize("shape", [(1, 37, 53), (2, 24, 40)])
@pytest.mark.parametrize("path", [0, DIRECT])
def test_first_conv_8bit_rgb_7x7_s2_bit_exact(shape, path):
    """The network's first conv (config 3): 8-bit unsigned image codes with 3 channels,
    7x7 stride 2 padding 3, 4-bit weight values (stored as 8-bit codes: a 3-channel row has
    no 4-bit packed layout), 64 channels of 4-bit codes out. The automatic choice is the F16
    tensor-core stem kernel; forcing path 2 runs the exact int32 CUDA-core kernel."""
    n, h, wd = shape
    rng = np.random.default_rng(h * 1000 + wd)
    x = synth.act_codes(rng, (n, h, wd, 3), 8)
    w = synth.weight_codes(rng, (64, 7, 7, 3), 4, "normal2")
    std = np.sqrt(147 * np.mean(np.arange(256) ** 2) * 4.0)
    m0, sh, b = _params(rng, 1, 64, 4, calib_std=std)
    got, want, used = conv_pair(x, 8, w, 8, stride=2, pad=3, out_bits=4, m0=m0, shift=sh, bias=b, path=path)
    assert used == (STEM if path == 0 else DIRECT)
    assert_same(got, want, 64, 4, f"first conv {shape}")
    assert len(np.unique(oracle_unpack(want, 64, 4))) > 4


# (n, h, w, cout, out_bits, stride, pad, levels, level, w_lim, calibrated): the stem kernel's
# output widths, channel counts (one and several 32-column groups, a 16-column tail with
# int32 out), geometries whose receptive fields leave the image on every side, a tile count
# that is not a multiple of the SM count, per-level tables, 7-bit weights, and requant shifts
# that force the int64 epilogue
STEM_CASES = [
    (1, 29, 31, 64, 2, 2, 3, 1, 0, 7, True),
    (2, 17, 45, 32, 3, 1, 3, 1, 0, 7, True),
    (1, 40, 40, 96, 8, 2, 0, 3, 2, 7, True),
    (3, 23, 19, 48, 32, 2, 3, 1, 0, 7, True),
    (1, 64, 90, 256, 4, 2, 3, 2, 1, 21, True),
    (1, 16, 16, 64, 4, 1, 1, 1, 0, 7, False),
    (1, 7, 7, 16, 32, 1, 0, 1, 0, 7, True),
]


@pytest.mark.parametrize("case", STEM_CASES, ids=[str(i) for i in range(len(STEM_CASES))])
def test_stem_kernel_bit_exact(case):
    n, h, wd, cout, out_bits, stride, pad, levels, level, w_lim, calibrated = case
    rng = np.random.default_rng(1000 + h * wd + cout)
    x = synth.act_codes(rng, (n, h, wd, 3), 8)
    w = rng.integers(-w_lim, w_lim + 1, size=(cout, 7, 7, 3)).astype(np.int32)
    std = np.sqrt(147 * np.mean(np.arange(256) ** 2) * np.mean(np.arange(-w_lim, w_lim + 1) ** 2))
    if out_bits == 32:
        m0 = sh = None
        b = rng.integers(-5000, 5000, size=(levels, cout)).astype(np.int32)
    elif calibrated:
        m0, sh, b = _params(rng, levels, cout, out_bits, calib_std=std)
    else:
        m0, sh, b = _params(rng, levels, cout, out_bits)
        sh[:, ::3] = 1  # R = 32: outside the 32-bit fast form
        sh[:, 1::5] = -4
    got, want, used = conv_pair(x, 8, w, 8, stride=stride, pad=pad, out_bits=out_bits, m0=m0, shift=sh, bias=b,
                                level=level)
    assert used == STEM
    assert_same(got, want, cout, out_bits, f"stem {case}")


def test_first_conv_full_size_bit_exact():
    """The first conv at the config-3 size (batch 8, 800x1344 after padding), on the F16 stem
    kernel: every output byte against the oracle's full convolution (about 40 GOP)."""
    import oracle
    import torch
    from gpu_util import dev
    from paper_2007_06919_gb300 import aqd
    rng = np.random.default_rng(3)
    n, h, wd = 8, 800, 1344
    x = synth.act_codes(rng, (n, h, wd, 3), 8)
    w = synth.weight_codes(rng, (64, 7, 7, 3), 4, "normal2")
    std = np.sqrt(147 * np.mean(np.arange(256) ** 2) * 4.0)
    m0, sh, b = _params(rng, 1, 64, 4, calib_std=std)
    xt = oracle.CodeTensor.from_codes(x, 8)
    W, wp = weights(w, 8)
    X = aqd.DTensor(dev(xt.packed), n, h, wd, 3, 8)
    Y = aqd.DTensor.empty(n, 400, 672, 64, 4)
    Y.data.fill_(0xA5)
    aqd.conv_int(X, W, 2, 3, Y, rq=aqd.RequantParams.from_numpy(m0, sh, b))
    assert aqd.last_conv_path() == STEM
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    want = oracle.conv_int(xt, wp, 8, 0, 7, 7, 2, 3, 64, m0=m0, shift=sh, bias=b, out_bits=4)
    assert_same(Y.data.cpu().numpy().reshape(want.packed.shape), want.packed, 64, 4, "stem, full size")


def oracle_unpack(packed, c, bits):
    import oracle
    return oracle.unpack(packed, c, bits)


# (x_bits, w_bits, n, h, w, cin, cout, out_bits): 8-bit operands on the tensor cores, split
# into 4-bit halves (activation planes x_lo, 16 x_hi; weight rows w_lo, w_hi)
WIDE_CASES = [
    (8, 4, 2, 11, 13, 128, 64, 4),     # 8-bit activations, 4-bit weights: two planes
    (8, 8, 1, 9, 17, 256, 256, 8),     # both 8-bit: two planes, split weights
    (2, 8, 2, 7, 9, 128, 96, 2),       # 8-bit weights only
    (4, 8, 1, 12, 10, 256, 80, 32),    # int32 output
    (8, 8, 3, 5, 6, 128, 384, 4),      # three 128-channel output blocks
]


@pytest.mark.parametrize("case", WIDE_CASES, ids=[str(i) for i in range(len(WIDE_CASES))])
@pytest.mark.parametrize("pairs", [True, False])
def test_wide_operands_on_tensor_cores_bit_exact(case, pairs):
    xb, wb, n, h, wd, cin, cout, ob = case
    rng = np.random.default_rng(hash(case) % 2 ** 32 + 7)
    x = synth.act_codes(rng, (n, h, wd, cin), xb)
    w = rng.integers(-(1 << (wb - 1)), 1 << (wb - 1), size=(cout, 3, 3, cin)).astype(np.int32)
    std = np.sqrt(9 * cin * np.mean(np.arange(1 << xb) ** 2) * (1 << (2 * wb - 2)) / 3)
    m0, sh, b = _params(rng, 1, cout, ob if ob != 32 else 4, calib_std=std)
    got, want, used = conv_pair(x, xb, w, wb, out_bits=ob, m0=m0, shift=sh, bias=b,
                                path=TC if pairs else TC_NO_PAIR, workspace=True)
    assert used == (4 if pairs else 3)
    assert_same(got, want, cout, ob, f"wide case {case}")


def test_wide_operands_exact_at_the_bound():
    """Every code 255 and every weight -128 or 127 (signs mixed per channel), K = 3456 (the
    FP32 partial sums D1 <= 3825 K stay below 2^24): int32 outputs equal the oracle's."""
    cin = 384
    x = np.full((1, 4, 5, cin), 255, np.int32)
    w = np.full((64, 3, 3, cin), -128, np.int32)
    w[1::2] = 127
    w[3, :, :, ::2] = -1
    got, want, used = conv_pair(x, 8, w, 8, pad=1, out_bits=32, bias=np.zeros((1, 64), np.int32), path=TC,
                                workspace=True)
    assert used == 4
    assert_same(got, want, 64, 32, "wide exactness")
    assert np.abs(want.view(np.int32)).max() > (1 << 26)


@pytest.mark.parametrize("neg_m0", [False, True])
@pytest.mark.parametrize("pairs", [True, False])
def test_two_bit_requant_edges(neg_m0, pairs):
    """2-bit outputs on the workspace path at the edges of Eq. 2's rescale: total shifts
    R = 31 + shift from 1 to 62 (both the 32-bit form, R >= 33, and the int64 form in one
    tile), biases up to +-2^29 (codes pinned at 0 or 3 for many channels), and negative
    multipliers in some channels."""
    rng = np.random.default_rng(11 + 2 * neg_m0 + pairs)
    n, h, wd, cin, cout = 2, 9, 13, 256, 256
    x = synth.act_codes(rng, (n, h, wd, cin), 2)
    w = synth.weight_codes(rng, (cout, 3, 3, cin), 2)
    m0 = rng.integers(1 << 30, 1 << 31, size=(1, cout), dtype=np.int64).astype(np.int32)
    sh = rng.integers(-30, 32, size=(1, cout)).astype(np.int8)
    sh[0, :64] = rng.integers(4, 8, size=64)         # a band where codes spread over 0..3
    b = rng.integers(-(1 << 29), 1 << 29, size=(1, cout)).astype(np.int32)
    b[0, :64] = rng.integers(-40, 40, size=64)
    if neg_m0:
        m0[0, ::7] = -m0[0, ::7]
    got, want, used = conv_pair(x, 2, w, 2, out_bits=2, m0=m0, shift=sh, bias=b,
                                path=TC if pairs else TC_NO_PAIR, workspace=True)
    assert used == (4 if pairs else 3)
    assert_same(got, want, cout, 2, "2-bit requant edges")
    codes = oracle_unpack(want, cout, 2)
    assert len(np.unique(codes[..., :64])) == 4


@pytest.mark.parametrize("out_bits", [2, 3, 4, 8])
@pytest.mark.parametrize("pairs", [True, False])
def test_k_bit_requant_edges(out_bits, pairs):
    """Eq. 2's clip at both ends for every code width on the workspace path, in the 32-bit
    requant form (every R = 31 + shift >= 40 - k here). A band of channels sits at the
    smallest of those R with biases that spread the codes over the whole range and past
    both ends of the clip; the others take R up to 62, biases up to +-2^29 and some
    negative multipliers."""
    rng = np.random.default_rng(40 + out_bits + 10 * pairs)
    n, h, wd, cin, cout = 2, 9, 13, 256, 256
    x = synth.act_codes(rng, (n, h, wd, cin), 2)
    w = synth.weight_codes(rng, (cout, 3, 3, cin), 2)
    qmax = (1 << out_bits) - 1
    r_min = 40 - out_bits
    m0 = rng.integers(1 << 30, 1 << 31, size=(1, cout), dtype=np.int64).astype(np.int32)
    sh = rng.integers(r_min - 31, 32, size=(1, cout)).astype(np.int8)
    b = rng.integers(-(1 << 29), 1 << 29, size=(1, cout)).astype(np.int32)
    band = slice(0, 96)
    m0[0, band] = rng.integers((1 << 31) - 4096, 1 << 31, size=96)
    sh[0, band] = r_min - 31 + rng.integers(0, 2, size=96)
    step = 1 << (9 - out_bits)            # accumulator units per code at R = r_min
    b[0, band] = rng.integers(-300, (qmax + 1) * step + 300, size=96)
    m0[0, 96::7] = -m0[0, 96::7]
    got, want, used = conv_pair(x, 2, w, 2, out_bits=out_bits, m0=m0, shift=sh, bias=b,
                                path=TC if pairs else TC_NO_PAIR, workspace=True)
    assert used == (4 if pairs else 3)
    assert_same(got, want, cout, out_bits, f"{out_bits}-bit requant edges")
    codes = oracle_unpack(want, cout, out_bits)[..., band]
    assert codes.min() == 0 and codes.max() == qmax
    assert len(np.unique(codes)) == qmax + 1 if out_bits <= 4 else len(np.unique(codes)) > 100
