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


# 16-byte units (4-bit 64 / 96 ch, 2-bit 256 ch, 8-bit 32 ch), single words (2-bit 32 ch: 8-byte
# rows; 8-bit 4 ch), and the generic kernel (8-bit 3 ch, 3-bit)
@pytest.mark.parametrize("bits,c,k,stride,pad", [(4, 64, 3, 2, 1), (2, 256, 3, 2, 1), (8, 3, 2, 2, 0),
                                                  (3, 32, 3, 1, 1), (2, 32, 3, 1, 1), (8, 32, 3, 2, 1),
                                                  (8, 4, 2, 2, 0), (4, 96, 3, 2, 0)])
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
