"""The FP4 tensor-core pipe for 2-bit codes (tcgen05 kind::mxf4nvf4 with unit UE8M0 block
scales): a code n and a weight w are the E2M1 values n / 2 and w / 2 (|w| <= 4), so each
product is an exact integer / 4 and the FP32 accumulator holds the exact sum / 4. Every
output is compared byte for byte with the oracle and with the same call on the E4M3 pipe,
on CTA pairs and on single CTAs, for the weight formats and widths the pipe takes, every
output width, code and int32 skips (Eq. 7, both directions, 2x up-read), grouped levels with
per-level tables (multi-level BN), and ragged and degenerate shapes."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_same, conv_pair, to_device, weights
from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu

FP4, TC, TC_NO_PAIR, TC_NO_FP4, TC_NO_PAIR_NO_FP4 = 6, 1, 3, 4, 5


def _w(rng, wb, fmt, shape):
    if fmt == 0:
        return rng.integers(-(1 << (wb - 1)), 1 << (wb - 1), size=shape).astype(np.int32)
    return rng.integers(0, 1 << wb, size=shape).astype(np.int32)


# (n, h, w, cin, cout, w_bits, w_format, out_bits)
CASES = [
    (2, 11, 9, 256, 80, 2, 0, 32),     # int32 heads, N tile 80
    (1, 13, 21, 256, 96, 2, 0, 2),     # 2-bit codes out, ragged rows
    (2, 7, 30, 512, 128, 3, 0, 4),     # 3-bit weights (|w| <= 4), two chunks per tap
    (1, 9, 13, 256, 64, 2, 1, 2),      # Eq. 3 odd weights (+-1, +-3)
    (2, 5, 7, 256, 240, 2, 0, 32),     # widest N tile the pipe takes (two accumulators + scales)
    (2, 6, 9, 256, 224, 2, 0, 3),      # 3-bit codes out
    (1, 1, 1, 256, 32, 2, 0, 2),       # 1x1 image: every tap but the centre pads
    (3, 4, 37, 256, 16, 3, 0, 8),      # 16 channels, 8-bit codes out
]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
@pytest.mark.parametrize("pairs", [True, False])
def test_fp4_matches_oracle_and_e4m3(case, pairs):
    n, h, wd, cin, cout, wb, fmt, ob = case
    rng = np.random.default_rng(hash(case) % 2 ** 32 + 17)
    x = synth.act_codes(rng, (n, h, wd, cin), 2)
    w = _w(rng, wb, fmt, (cout, 3, 3, cin))
    max_w = (1 << (wb - 1)) if fmt == 0 else (1 << wb) - 1
    std = np.sqrt(9 * cin * np.mean(np.arange(4) ** 2) * max_w ** 2 / 3)
    m0, sh, b = synth.requant_params(rng, 1, cout, calib_std=std, out_bits=ob if ob != 32 else 4)
    wp = weights(w, wb, fmt)
    got, want, used = conv_pair(x, 2, w, wb, w_format=fmt, out_bits=ob, m0=m0, shift=sh, bias=b,
                                path=TC if pairs else TC_NO_PAIR, workspace=True, wprep=wp)
    assert used == FP4
    assert_same(got, want, cout, ob, f"fp4 case {case}")
    e4, _, used8 = conv_pair(x, 2, w, wb, w_format=fmt, out_bits=ob, m0=m0, shift=sh, bias=b,
                             path=TC_NO_FP4 if pairs else TC_NO_PAIR_NO_FP4, workspace=True, wprep=wp)
    assert used8 == (4 if pairs else 3)
    assert np.array_equal(got, e4)


@pytest.mark.parametrize("skip_bits,upsample,mirror", [(2, 1, 0), (4, 1, 1), (32, 2, 0), (32, 1, 1), (2, 2, 0)])
def test_fp4_with_skip(skip_bits, upsample, mirror):
    """Eq. 7 in the epilogue of the FP4 pipe: code and int32 skips, both directions, 2x up-read."""
    rng = np.random.default_rng(70 + skip_bits + 10 * upsample + mirror)
    n, h, wd, cin, cout = 2, 10, 13, 256, 128
    x = synth.act_codes(rng, (n, h, wd, cin), 2)
    w = synth.weight_codes(rng, (cout, 3, 3, cin), 2)
    m0, sh, b = synth.requant_params(rng, 1, cout, calib_std=60.0, out_bits=2)
    sh_ = (h + upsample - 1) // upsample, (wd + upsample - 1) // upsample
    if skip_bits == 32:
        skip = rng.integers(-300, 300, size=(n, sh_[0], sh_[1], cout)).astype(np.int32)
    else:
        skip = synth.act_codes(rng, (n, sh_[0], sh_[1], cout), skip_bits)
    c, d = synth.skip_params(rng, 1, cout, sh)
    got, want, used = conv_pair(x, 2, w, 2, out_bits=2, m0=m0, shift=sh, bias=b, skip=skip, skip_bits=skip_bits,
                                skip_c=c, skip_d=d, upsample=upsample, scale_main=mirror, path=TC, workspace=True)
    assert used == FP4
    assert_same(got, want, cout, 2, "fp4 skip")


def test_fp4_exact_at_large_sums():
    """Every code 3 and weights of one sign per channel (3-bit, |w| = 4 and 3), cin 2048
    (K = 18432): sums reach 221,184 in magnitude, 2^17.8; int32 outputs equal the oracle's."""
    cin, cout = 2048, 32
    x = np.full((1, 4, 5, cin), 3, np.int32)
    rng = np.random.default_rng(9)
    x[0, 1, 2, ::5] = rng.integers(0, 4, size=x[0, 1, 2, ::5].shape)
    w = np.full((cout, 3, 3, cin), -4, np.int32)
    w[1::2] = 3
    w[7, :, :, ::2] = 1
    got, want, used = conv_pair(x, 2, w, 3, out_bits=32, bias=np.zeros((1, cout), np.int32), path=TC,
                                workspace=True)
    assert used == FP4
    assert_same(got, want, cout, 32, "fp4 exactness")
    assert np.abs(want.view(np.int32)).max() > (1 << 17)


def test_fp4_grouped_levels_bit_exact():
    """The head's fused 256->84 output conv over five FPN levels in one grouped launch with a
    bias row per level (multi-level BN), on the FP4 pipe."""
    levels = [(20, 34), (10, 17), (5, 9), (3, 5), (2, 3)]
    wl = synth.head_tower(12, 2, 2, levels=levels, calibrated=True)
    cls, box = wl.convs[4:]
    w = np.concatenate([cls.w, box.w])
    bias = np.concatenate([cls.bias, box.bias], axis=1)
    W, wp = weights(w, 2)
    xts = [oracle.CodeTensor.from_codes(x, 2) for x in wl.inputs]
    xs = [to_device(t) for t in xts]
    ys = [aqd.DTensor.empty(t.n, t.h, t.w, 84, 32) for t in xts]
    jobs = [(xs[l], ys[l], None, l) for l in range(5)]
    aqd.conv_int_grouped(jobs, W, 1, 1, rq=aqd.RequantParams.from_numpy(None, None, bias),
                         workspace=aqd.workspace_for(jobs, W, 1, 1))
    assert aqd.last_conv_path() == FP4
    torch.cuda.synchronize()
    for l in range(5):
        want = oracle.conv_int(xts[l], wp, 2, 0, 3, 3, 1, 1, 84, level=l, bias=bias, levels=5, out_bits=32)
        assert_same(ys[l].data.cpu().numpy().reshape(want.packed.shape), want.packed, 84, 32, f"level {l}")
    assert aqd.device_status() == 0


@pytest.mark.parametrize("shape", [(1, 1, 1), (2, 3, 300), (1, 37, 2), (3, 7, 11)])
def test_fp4_edge_shapes(shape):
    """Tiles that cross image rows and images, 1x1 and single-column images, on the nibble image."""
    n, h, wd = shape
    rng = np.random.default_rng(n * 1000 + h * 10 + wd + 5)
    x = synth.act_codes(rng, (n, h, wd, 256), 2)
    w = synth.weight_codes(rng, (96, 3, 3, 256), 2)
    m0, sh, b = synth.requant_params(rng, 1, 96, calib_std=37.0, out_bits=2)
    got, want, used = conv_pair(x, 2, w, 2, out_bits=2, m0=m0, shift=sh, bias=b, path=TC, workspace=True)
    assert used == FP4
    assert_same(got, want, 96, 2, f"fp4 edge {shape}")
