"""aqd_conv_int_static_workspace: the workspace-path convolution on the library's own fixed
workspace, allocating nothing. Two calls in a row (the second on different inputs, so a
stale workspace would show) must give the same bytes as aqd_conv_int with a caller
workspace; a problem larger than the fixed workspace is refused before any launch.
(Named to be collected last; it passes alone and after the other tests.)"""
import numpy as np
import pytest

from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu


def _case(seed, n, h, w, cin, cout, bits):
    import torch
    rng = np.random.default_rng(seed)
    x = synth.act_codes(rng, (n, h, w, cin), bits)
    wc = synth.weight_codes(rng, (cout, 3, 3, cin), bits)
    m0, sh, b = synth.requant_params(rng, 1, cout, calib_std=40.0, out_bits=bits)
    X = aqd.DTensor.from_codes(torch.from_numpy(x).cuda(), bits)
    W = aqd.ConvWeights(torch.from_numpy(wc).cuda(), bits)
    rq = aqd.RequantParams.from_numpy(m0, sh, b)
    return X, W, rq


def test_two_calls_match_the_workspace_entry_point():
    import torch
    for seed, shape in ((1, (2, 13, 21, 256, 256, 2)), (2, (1, 9, 30, 128, 96, 4))):
        n, h, w, cin, cout, bits = shape
        X, W, rq = _case(seed, n, h, w, cin, cout, bits)
        ref = aqd.DTensor.empty(n, h, w, cout, bits)
        ws = aqd.workspace_for([(X, ref, None, 0)], W, 1, 1)
        aqd.conv_int(X, W, 1, 1, ref, rq=rq, workspace=ws)
        got = aqd.DTensor.empty(n, h, w, cout, bits)
        got.data.fill_(0xA5)
        aqd.conv_int_static_workspace(X, W, 1, 1, got, rq=rq)
        assert aqd.last_conv_path() in (3, 4)
        torch.cuda.synchronize()
        assert torch.equal(got.data, ref.data), f"call with seed {seed}"
    assert aqd.device_status() == 0


def test_too_large_for_the_static_workspace_is_refused():
    import torch
    # 4 x 100 x 168 x 256 bytes of expanded input > 16 MiB
    X = aqd.DTensor.empty(4, 100, 168, 256, 2)
    Y = aqd.DTensor.empty(4, 100, 168, 256, 2)
    rng = np.random.default_rng(0)
    W = aqd.ConvWeights(torch.from_numpy(synth.weight_codes(rng, (256, 3, 3, 256), 2)).cuda(), 2)
    rq = aqd.RequantParams.from_numpy(np.full((1, 256), 1 << 30), np.full((1, 256), 8), np.zeros((1, 256)))
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int_static_workspace(X, W, 1, 1, Y, rq=rq)
    assert e.value.status == 2
    torch.cuda.synchronize()


def test_calls_off_the_workspace_path_are_refused():
    """8-bit activation codes with a skip run on the CUDA-core kernel, which reads no
    workspace, so the no-allocation entry point refuses them (AQD_ERR_UNSUPPORTED) instead
    of running a kernel that ignores its workspace; a forced CUDA-core path is refused the
    same way; an argument error is reported as AQD_ERR_INVALID, as aqd_conv_int reports it."""
    import torch
    rng = np.random.default_rng(3)
    n, h, w, c = 1, 6, 7, 128
    X = aqd.DTensor.from_codes(torch.from_numpy(synth.act_codes(rng, (n, h, w, c), 8)).cuda(), 8)
    S = aqd.DTensor.from_codes(torch.from_numpy(synth.act_codes(rng, (n, h, w, c), 8)).cuda(), 8)
    W = aqd.ConvWeights(torch.from_numpy(synth.weight_codes(rng, (c, 3, 3, c), 4)).cuda(), 4)
    m0, sh, b = synth.requant_params(rng, 1, c, calib_std=3000.0, out_bits=8)
    rq = aqd.RequantParams.from_numpy(m0, sh, b)
    cc, dd = synth.skip_params(rng, 1, c, sh)
    sp = aqd.SkipParams.from_numpy(cc, dd)
    Y = aqd.DTensor.empty(n, h, w, c, 8)
    Y.data.fill_(0x5A)
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int_static_workspace(X, W, 1, 1, Y, rq=rq, skip=S, sp=sp)
    assert e.value.status == 2
    # the same call through aqd_conv_int (no workspace needed) runs, so the refusal is the
    # entry point's own rule, not an unsupported convolution
    aqd.conv_int(X, W, 1, 1, aqd.DTensor.empty(n, h, w, c, 8), rq=rq, skip=S, sp=sp)
    # a forced CUDA-core path is refused as well, even where the workspace path applies
    X2, W2, rq2 = _case(4, 1, 5, 9, 128, 64, 2)
    Y2 = aqd.DTensor.empty(1, 5, 9, 64, 2)
    old = aqd.set_conv_path(2)
    try:
        with pytest.raises(aqd.AqdError) as e:
            aqd.conv_int_static_workspace(X2, W2, 1, 1, Y2, rq=rq2)
        assert e.value.status == 2
    finally:
        aqd.set_conv_path(old)
    # weights for 64 input channels on a 128-channel input: an argument error
    W3 = aqd.ConvWeights(torch.from_numpy(synth.weight_codes(rng, (64, 3, 3, 64), 2)).cuda(), 2)
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int_static_workspace(X2, W3, 1, 1, Y2, rq=rq2)
    assert e.value.status == 1
    torch.cuda.synchronize()
    # nothing was launched into the refused calls' outputs
    assert bool((Y.data == 0x5A).all())
    assert aqd.device_status() == 0
