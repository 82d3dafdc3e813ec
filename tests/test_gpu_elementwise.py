"""GPU parity of the element-wise ops against the oracle: packing, requant (Eq. 6 + Eq. 2),
the standalone skip add (Eq. 7/8, FPN upsample read), max-pooling on codes (Sec. 3.2.4)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_same, dev, to_device
from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("bits,c", [(2, 64), (3, 96), (4, 256), (8, 32), (8, 3), (8, 80)])
def test_pack_unpack_match_oracle(bits, c):
    rng = np.random.default_rng(bits * 100 + c)
    codes = rng.integers(0, 1 << bits, size=(517, c)).astype(np.int32)
    packed = aqd.pack_codes(dev(codes), bits)
    torch.cuda.synchronize()
    assert np.array_equal(packed.cpu().numpy(), oracle.pack(codes, bits))
    back = aqd.unpack_codes(dev(oracle.pack(codes, bits)), c, bits)
    assert np.array_equal(back.cpu().numpy(), codes)
    signed = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(33, c)).astype(np.int32)
    back = aqd.unpack_codes(dev(oracle.pack(signed, bits)), c, bits, signed=True)
    assert np.array_equal(back.cpu().numpy(), signed)


@pytest.mark.parametrize("out_bits,c,levels,level", [(2, 256, 5, 3), (3, 64, 1, 0), (4, 128, 2, 1), (8, 64, 1, 0),
                                                      (32, 80, 5, 4)])
def test_requant_matches_oracle(out_bits, c, levels, level):
    rng = np.random.default_rng(out_bits * 7 + c)
    acc = rng.integers(-40000, 40000, size=(2, 37, 29, c)).astype(np.int32)
    acc[0, 0, 0, :4] = (2 ** 31 - 1, -2 ** 31, 2 ** 31 - 5, -7)
    m0, sh, b = synth.requant_params(rng, levels, c, calib_std=20000.0, out_bits=min(out_bits, 8))
    ref = oracle.requant(oracle.CodeTensor.from_codes(acc, 32), m0, sh, b, level=level, levels=levels,
                         out_bits=out_bits)
    A = to_device(oracle.CodeTensor.from_codes(acc, 32))
    Y = aqd.DTensor.empty(2, 37, 29, c, out_bits)
    aqd.requant(A, aqd.RequantParams.from_numpy(m0, sh, b), Y, level=level)
    torch.cuda.synchronize()
    assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, c, out_bits, "requant")


@pytest.mark.parametrize("shape,out_bits,shift_range", [
    ((4, 100, 168, 256), 2, (8, 20)),       # many units per thread (the blocks stride), 32-bit form
    ((2, 13, 21, 256), 4, (-31, 31)),       # R = 0 .. 62 in one table: the int64 form
    ((1, 9, 7, 1056), 2, (8, 20)),          # more channels than the staged table holds
    ((3, 5, 11, 512), 8, (-3, 31)),         # exactly the staged-table limit, some R < 33
    ((2, 17, 23, 96), 3, (8, 20))])         # 3 channel groups: a warp spans several groups
def test_requant_forms_and_sizes(shape, out_bits, shift_range):
    """aqd_requant's forms: the 32-bit form (every R >= 33) over a tensor with several units per
    thread, the int64 form when some R < 33, the per-element table path past the staged
    channel limit, and int32 extremes that saturate Eq. 6's sum before the multiply. The
    int32 input goes through the shared-memory staging of whole 256-unit spans and of a
    partial last span."""
    n, h, w, c = shape
    rng = np.random.default_rng(sum(shape) + out_bits)
    acc = rng.integers(-30000, 30000, size=shape).astype(np.int32)
    acc[0, 0, 0, :6] = (2 ** 31 - 1, -2 ** 31, 2 ** 31 - 5, -7, 2 ** 30, -2 ** 30)
    m0 = rng.integers(1 << 30, 1 << 31, size=(1, c), dtype=np.int64).astype(np.int32)
    m0[0, ::5] = -m0[0, ::5]
    sh = rng.integers(shift_range[0], shift_range[1] + 1, size=(1, c)).astype(np.int8)
    b = rng.integers(-(1 << 30), 1 << 30, size=(1, c)).astype(np.int32)
    b[0, : c // 2] = rng.integers(-3000, 3000, size=c // 2)
    ref = oracle.requant(oracle.CodeTensor.from_codes(acc, 32), m0, sh, b, level=0, levels=1, out_bits=out_bits)
    Y = aqd.DTensor.empty(n, h, w, c, out_bits)
    Y.data.fill_(0xA5)
    aqd.requant(to_device(oracle.CodeTensor.from_codes(acc, 32)), aqd.RequantParams.from_numpy(m0, sh, b), Y)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, c, out_bits, f"requant {shape}")
    codes = oracle.unpack(ref.packed, c, out_bits)
    assert codes.min() == 0 and codes.max() == (1 << out_bits) - 1


@pytest.mark.parametrize("a_bits,b_bits,up,mirror,out_bits,with_rq",
                         [(32, 4, 1, 0, 4, True), (4, 4, 1, 1, 4, True), (32, 32, 2, 0, 2, True),
                          (2, 8, 2, 1, 32, False), (32, 3, 1, 0, 32, True), (8, 4, 1, 0, 3, True)])
def test_residual_add_matches_oracle(a_bits, b_bits, up, mirror, out_bits, with_rq):
    rng = np.random.default_rng(a_bits + 3 * b_bits + 11 * up + 101 * mirror)
    n, h, w, c = 2, 25, 42, 64
    a = (rng.integers(-30000, 30000, size=(n, h, w, c)) if a_bits == 32 else
         synth.act_codes(rng, (n, h, w, c), a_bits)).astype(np.int32)
    bh, bw = (h + up - 1) // up, (w + up - 1) // up
    b = (rng.integers(-30000, 30000, size=(n, bh, bw, c)) if b_bits == 32 else
         synth.act_codes(rng, (n, bh, bw, c), b_bits)).astype(np.int32)
    m0, sh, bias = synth.requant_params(rng, 1, c, calib_std=20000.0, out_bits=min(out_bits, 8))
    cc, dd = synth.skip_params(rng, 1, c, sh)
    kw = dict(m0=m0, shift=sh, bias=bias) if with_rq else {}
    at, bt = oracle.CodeTensor.from_codes(a, a_bits), oracle.CodeTensor.from_codes(b, b_bits)
    ref = oracle.residual_add(at, bt, cc, dd, upsample=up, scale_a=mirror, out_bits=out_bits, **kw)
    Y = aqd.DTensor.empty(n, h, w, c, out_bits)
    rq = aqd.RequantParams.from_numpy(m0, sh, bias) if with_rq else None
    aqd.residual_add_int(to_device(at), to_device(bt), aqd.SkipParams.from_numpy(cc, dd, up, mirror), Y, rq=rq)
    torch.cuda.synchronize()
    assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, c, out_bits, "residual")


@pytest.mark.parametrize("with_rq,mirror", [(False, 0), (True, 1)])
def test_residual_add_int32_spans(with_rq, mirror):
    """The skip add with an int32 main operand over more units than one pass of the grid
    (blocks take several 256-unit spans, the last one partial), a 2x-upsampled 4-bit skip,
    and an int32 result staged back through shared memory (without rq) or 4-bit codes."""
    rng = np.random.default_rng(77 + mirror)
    n, h, w, c = 8, 100, 167, 64
    a = rng.integers(-(1 << 30), 1 << 30, size=(n, h, w, c)).astype(np.int32)
    a[0, 0, 0, :4] = (2 ** 31 - 1, -2 ** 31, 2 ** 31 - 2, -2 ** 31 + 1)
    b = synth.act_codes(rng, (n, (h + 1) // 2, (w + 1) // 2, c), 4)
    m0, sh, bias = synth.requant_params(rng, 1, c, calib_std=2.0 ** 29, out_bits=4)
    cc = rng.integers(1 << 30, 1 << 31, size=(1, c), dtype=np.int64).astype(np.int32)
    dd = rng.integers(4, 12, size=(1, c)).astype(np.int8)
    out_bits = 4 if with_rq else 32
    kw = dict(m0=m0, shift=sh, bias=bias) if with_rq else {}
    at, bt = oracle.CodeTensor.from_codes(a, 32), oracle.CodeTensor.from_codes(b, 4)
    ref = oracle.residual_add(at, bt, cc, dd, upsample=2, scale_a=mirror, out_bits=out_bits, **kw)
    Y = aqd.DTensor.empty(n, h, w, c, out_bits)
    Y.data.fill_(0xA5)
    rq = aqd.RequantParams.from_numpy(m0, sh, bias) if with_rq else None
    aqd.residual_add_int(to_device(at), to_device(bt), aqd.SkipParams.from_numpy(cc, dd, 2, mirror), Y, rq=rq)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, c, out_bits, "residual spans")


@pytest.mark.parametrize("c,b_bits,out_bits,wide", [(256, 2, 2, True), (256, 4, 4, True), (256, 8, 32, True),
                                                     (128, 4, 8, False), (128, 4, 8, True), (64, 4, 2, False),
                                                     (96, 8, 4, True), (32, 2, 2, False)])
def test_residual_add_int32_lane_forms(c, b_bits, out_bits, wide):
    """The int32 skip add's two exact forms side by side: channels 0 .. c/2 - 1 take skip
    constants at the edge of the 32-bit form (s c + 2^(d-1) at the widest code s equal to
    2^31 - 1, and a bias whose sum with rhu(s c, d) reaches +-(2^31 - 1) exactly), the other
    half one channel with a skip multiplier too wide for it (its warp runs the int64 form);
    accumulators at the int32 extremes saturate Eq. 6's sum. 4, 2 and 1 channels per lane."""
    rng = np.random.default_rng(c * 7 + b_bits + out_bits)
    n, h, w = 2, 19, 23
    a = rng.integers(-(1 << 31), 1 << 31, size=(n, h, w, c), dtype=np.int64).astype(np.int32)
    a[0, 0, :3, :] = np.array([2 ** 31 - 1, -2 ** 31, 0], dtype=np.int64)[:, None].astype(np.int32)
    b = synth.act_codes(rng, (n, h, w, c), b_bits)
    b[0, 0, :2, :] = (1 << b_bits) - 1
    smax = (1 << b_bits) - 1
    dd = rng.integers(0, 12, size=(1, c)).astype(np.int8)
    half = np.where(dd > 0, 1 << np.maximum(dd.astype(np.int64) - 1, 0), 0)
    cc = np.zeros((1, c), dtype=np.int64)
    bias = rng.integers(-(1 << 20), 1 << 20, size=(1, c)).astype(np.int64)
    for j in range(c // 2):
        if j % 2 == 0:   # s c + half = 2^31 - 1 at s = smax, bias + rhu = 2^31 - 1
            cc[0, j] = (2 ** 31 - 1 - half[0, j]) // smax
            bias[0, j] = 2 ** 31 - 1 - ((smax * cc[0, j] + half[0, j]) >> int(dd[0, j]))
        else:            # s c + half >= -2^31, bias + rhu = -2^31
            cc[0, j] = -((2 ** 31 + half[0, j]) // smax)
            bias[0, j] = -2 ** 31 - ((smax * cc[0, j] + half[0, j]) >> int(dd[0, j]))
    cc[0, c // 2:] = rng.integers(-(1 << 12), 1 << 12, size=c - c // 2)
    if wide:
        cc[0, c - 1] = 2 ** 31 - 1   # too wide for the 32-bit form: this channel's warp takes int64
    cc, bias = cc.astype(np.int32), bias.astype(np.int32)
    m0 = rng.integers(1 << 30, 1 << 31, size=(1, c), dtype=np.int64).astype(np.int32)
    sh = rng.integers(20, 28, size=(1, c)).astype(np.int8)
    kw = dict(m0=m0, shift=sh, bias=bias) if out_bits != 32 else dict(bias=bias)
    at, bt = oracle.CodeTensor.from_codes(a, 32), oracle.CodeTensor.from_codes(b, b_bits)
    ref = oracle.residual_add(at, bt, cc, dd, upsample=1, scale_a=0, out_bits=out_bits, **kw)
    Y = aqd.DTensor.empty(n, h, w, c, out_bits)
    Y.data.fill_(0xA5)
    rq = aqd.RequantParams.from_numpy(m0, sh, bias) if out_bits != 32 else aqd.RequantParams.from_numpy(None, None, bias)
    aqd.residual_add_int(to_device(at), to_device(bt), aqd.SkipParams.from_numpy(cc, dd), Y, rq=rq)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, c, out_bits, "residual lane forms")


@pytest.mark.parametrize("c,a_bits,b_bits,out_bits", [(160, 4, 32, 2), (96, 8, 2, 32), (256, 3, 4, 4)])
def test_residual_add_packed_main_operand(c, a_bits, b_bits, out_bits):
    """The skip add with packed codes as the main operand (their bytes staged through shared
    memory as one range per span), channel counts whose group count divides the block
    (256) or not, and code, int32 or code outputs."""
    rng = np.random.default_rng(c + a_bits + b_bits)
    n, h, w = 3, 31, 45
    a = synth.act_codes(rng, (n, h, w, c), a_bits)
    b = (rng.integers(-8, 8, size=(n, h, w, c)) if b_bits == 32 else
         synth.act_codes(rng, (n, h, w, c), b_bits)).astype(np.int32)
    m0, sh, bias = synth.requant_params(rng, 1, c, calib_std=40.0, out_bits=min(out_bits, 8))
    cc, dd = synth.skip_params(rng, 1, c, sh)
    kw = dict(m0=m0, shift=sh, bias=bias) if out_bits != 32 else {}
    at, bt = oracle.CodeTensor.from_codes(a, a_bits), oracle.CodeTensor.from_codes(b, b_bits)
    ref = oracle.residual_add(at, bt, cc, dd, upsample=1, scale_a=0, out_bits=out_bits, **kw)
    Y = aqd.DTensor.empty(n, h, w, c, out_bits)
    Y.data.fill_(0xA5)
    rq = aqd.RequantParams.from_numpy(m0, sh, bias) if out_bits != 32 else None
    aqd.residual_add_int(to_device(at), to_device(bt), aqd.SkipParams.from_numpy(cc, dd), Y, rq=rq)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, c, out_bits, "residual packed main")


# 16-byte units (4-bit 64 / 96 ch, 2-bit 256 ch, 8-bit 32 ch), single words (2-bit 32 ch: 8-byte
# rows; 8-bit 4 ch), and the generic kernel (8-bit 3 ch, 3-bit)
@pytest.mark.parametrize("bits,c,k,stride,pad", [(4, 64, 3, 2, 1), (2, 256, 3, 2, 1), (8, 3, 2, 2, 0),
                                                  (3, 32, 3, 1, 1), (2, 32, 3, 1, 1), (8, 32, 3, 2, 1),
                                                  (8, 4, 2, 2, 0), (4, 96, 3, 2, 0), (4, 64, 3, 2, 2),
                                                  (2, 64, 3, 2, 1)])
def test_maxpool_matches_oracle(bits, c, k, stride, pad):
    rng = np.random.default_rng(bits + c)
    x = synth.act_codes(rng, (2, 41, 67, c), bits)
    xt = oracle.CodeTensor.from_codes(x, bits)
    ref = oracle.maxpool(xt, k, stride, pad)
    Y = aqd.DTensor.empty(ref.n, ref.h, ref.w, c, bits)
    aqd.maxpool_codes(to_device(xt), k, stride, pad, Y)
    torch.cuda.synchronize()
    assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, c, bits, "maxpool")


def test_device_status_is_clean():
    assert aqd.device_status() == 0


def test_staged_graph_replays_after_a_smaller_call():
    """A CUDA graph holding the staged skip add with a 256-channel table (the larger shared
    memory plan) still replays, bit-exact, after an eager call of the same kernel with a
    128-channel table: its shared-memory limit is never lowered below an earlier capture's."""
    rng = np.random.default_rng(314)

    def case(c, n=2, h=21, w=33):
        a = rng.integers(-30000, 30000, size=(n, h, w, c)).astype(np.int32)
        b = synth.act_codes(rng, (n, h, w, c), 4)
        m0, sh, bias = synth.requant_params(rng, 1, c, calib_std=20000.0, out_bits=2)
        cc, dd = synth.skip_params(rng, 1, c, sh)
        at, bt = oracle.CodeTensor.from_codes(a, 32), oracle.CodeTensor.from_codes(b, 4)
        ref = oracle.residual_add(at, bt, cc, dd, out_bits=2, m0=m0, shift=sh, bias=bias)
        args = (to_device(at), to_device(bt), aqd.SkipParams.from_numpy(cc, dd), aqd.DTensor.empty(n, h, w, c, 2),
                aqd.RequantParams.from_numpy(m0, sh, bias))
        return args, ref

    (a1, b1, s1, y1, r1), ref1 = case(256)
    (a2, b2, s2, y2, r2), ref2 = case(128)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        aqd.residual_add_int(a1, b1, s1, y1, rq=r1, stream=stream)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        aqd.residual_add_int(a1, b1, s1, y1, rq=r1, stream=stream)
    aqd.residual_add_int(a2, b2, s2, y2, rq=r2)
    torch.cuda.synchronize()
    y1.data.fill_(0xA5)
    g.replay()
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    assert_same(y1.data.cpu().numpy().reshape(ref1.packed.shape), ref1.packed, 256, 2, "graph replay")
    assert_same(y2.data.cpu().numpy().reshape(ref2.packed.shape), ref2.packed, 128, 2, "smaller call")
