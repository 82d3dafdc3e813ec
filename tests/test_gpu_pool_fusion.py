"""GPU parity of the max-pool fused into a convolution's expansion pass (aqd_maxpool_expand,
Sec. 3.2.4's max-pool on codes): the pooled codes against the oracle's max-pool, and the
pooled codes plus the byte image against the two separate calls (aqd_maxpool_codes, then
aqd_conv_expand_input), byte for byte; then the convolution read from the fused image against
the oracle's pool -> conv."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import to_device, weights
from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu


def _case(bits, c, n, h, w, k, stride, pad, seed):
    rng = np.random.default_rng(seed)
    x = oracle.CodeTensor.from_codes(synth.act_codes(rng, (n, h, w, c), bits), bits)
    ho, wo = aqd.conv_out_hw(h, w, k, k, stride, pad)
    wc = rng.integers(-2, 2, size=(64, 3, 3, c)).astype(np.int32)
    return rng, x, ho, wo, wc


@pytest.mark.parametrize("bits,c,n,h,w,k,stride,pad", [
    (4, 64, 2, 37, 51, 3, 2, 1),     # the stem pool, odd sizes (clamped taps on both far edges)
    (2, 64, 1, 40, 30, 3, 2, 1),     # 2-bit codes: 64 byte-image bytes per 16-byte unit
    (4, 192, 1, 9, 12, 3, 2, 0),     # no padding, 6 units per pixel (no power of two)
    (4, 128, 3, 26, 9, 3, 2, 2),     # padding 2: taps clamped twice
    (2, 256, 1, 8, 8, 3, 2, 1)])     # 4 units per pixel
def test_maxpool_expand_matches_separate_calls(bits, c, n, h, w, k, stride, pad):
    rng, x, ho, wo, wc = _case(bits, c, n, h, w, k, stride, pad, bits * 1000 + c + h)
    W, _ = weights(wc, 2)
    X = to_device(x)
    y_conv = aqd.DTensor.empty(n, ho, wo, 64, 32)
    Y1, Y2 = aqd.DTensor.empty(n, ho, wo, c, bits), aqd.DTensor.empty(n, ho, wo, c, bits)
    Y1.data.fill_(0xA5)
    Y2.data.fill_(0x5A)
    wsb = aqd.conv_workspace_bytes([(Y1, y_conv, None, 0)], W, 1, 1)
    assert wsb > 0
    ws1 = torch.full((wsb,), 0x11, dtype=torch.uint8, device="cuda")
    ws2 = torch.full((wsb,), 0x77, dtype=torch.uint8, device="cuda")
    aqd.maxpool_codes(X, k, stride, pad, Y1)
    aqd.conv_expand_input([(Y1, y_conv, None, 0)], W, 1, 1, ws1)
    aqd.maxpool_expand(X, k, stride, pad, Y2, W, 1, 1, ws2)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    ref = oracle.maxpool(x, k, stride, pad)
    assert np.array_equal(Y2.data.cpu().numpy().reshape(ref.packed.shape), ref.packed)
    assert torch.equal(Y1.data, Y2.data)
    assert torch.equal(ws1, ws2)


def test_conv_reads_the_fused_image():
    """pool -> conv with the pool in the expansion pass, against the oracle's pool then conv."""
    bits, c, n, h, w = 4, 64, 2, 45, 38
    rng, x, ho, wo, wc = _case(bits, c, n, h, w, 3, 2, 1, 99)
    W, wpk = weights(wc, 2)
    m0, sh, bias = synth.requant_params(rng, 1, 64, calib_std=60.0, out_bits=4)
    X = to_device(x)
    P = aqd.DTensor.empty(n, ho, wo, c, bits)
    Y = aqd.DTensor.empty(n, ho, wo, 64, 4)
    Y.data.fill_(0xA5)
    jobs = [(P, Y, None, 0)]
    ws = torch.empty(aqd.conv_workspace_bytes(jobs, W, 1, 1), dtype=torch.uint8, device="cuda")
    rq = aqd.RequantParams.from_numpy(m0, sh, bias)
    aqd.maxpool_expand(X, 3, 2, 1, P, W, 1, 1, ws)
    aqd.conv_int_grouped_expanded(jobs, W, 1, 1, rq=rq, workspace=ws)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    pooled = oracle.maxpool(x, 3, 2, 1)
    ref = oracle.conv_int(pooled, wpk, 2, 0, 3, 3, 1, 1, 64, m0=m0, shift=sh, bias=bias, out_bits=4)
    assert np.array_equal(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed)


def test_maxpool_expand_argument_errors():
    bits, c, n, h, w = 4, 64, 1, 16, 16
    rng, x, ho, wo, wc = _case(bits, c, n, h, w, 3, 2, 1, 5)
    W, _ = weights(wc, 2)
    X = to_device(x)
    P = aqd.DTensor.empty(n, ho, wo, c, bits)
    ws = torch.empty(aqd.conv_workspace_bytes([(P, aqd.DTensor.empty(n, ho, wo, 64, 32), None, 0)], W, 1, 1),
                     dtype=torch.uint8, device="cuda")
    with pytest.raises(aqd.AqdError) as e:          # 3-bit codes: no fused pool
        x3 = to_device(oracle.CodeTensor.from_codes(synth.act_codes(rng, (n, h, w, c), 3), 3))
        aqd.maxpool_expand(x3, 3, 2, 1, aqd.DTensor.empty(n, ho, wo, c, 3), W, 1, 1, ws)
    assert e.value.status == 2
    with pytest.raises(aqd.AqdError) as e:          # not a 3x3 stride-2 pool
        ho2, wo2 = aqd.conv_out_hw(h, w, 2, 2, 2, 0)
        aqd.maxpool_expand(X, 2, 2, 0, aqd.DTensor.empty(n, ho2, wo2, c, bits), W, 1, 1, ws)
    assert e.value.status == 2
    with pytest.raises(aqd.AqdError) as e:          # workspace too small for the conv
        aqd.maxpool_expand(X, 3, 2, 1, P, W, 1, 1, ws[:64])
    assert e.value.status == 2
    with pytest.raises(aqd.AqdError) as e:          # y not the pooled shape
        aqd.maxpool_expand(X, 3, 2, 1, aqd.DTensor.empty(n, ho + 1, wo, c, bits), W, 1, 1, ws)
    assert e.value.status == 1
    with pytest.raises(aqd.AqdError) as e:          # in place
        aqd.maxpool_expand(X, 1, 1, 0, X, W, 1, 1, ws)
    assert e.value.status == 1
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
