"""The device-side failure path of the tensor-core kernels, exercised without a fault: the
kernels' bounded mbarrier wait (shortened to 2 ms in a self-test kernel) waits on a barrier
that nobody arrives at, expires, latches AQD_ERR_TIMEOUT in the device status word and
raises the kernel's abort flag; a second role, waiting the full 1 s limit on another such
barrier, leaves through that flag. aqd_device_status then reports the timeout once and
clears it, and the context stays usable (a convolution right after is bit-exact)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import to_device, weights
from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu

TIMEOUT = 4  # AQD_ERR_TIMEOUT


def test_expired_wait_latches_timeout_and_unwinds():
    assert aqd.device_status() == 0
    out = torch.full((5,), -1, dtype=torch.int64, device="cuda")
    aqd.selftest_wait_timeout(out)
    torch.cuda.synchronize()
    r = out.cpu().tolist()
    assert r[4] == 1, "a barrier whose phase completed was not seen as complete"
    assert r[0] == 1, "the 2 ms wait did not expire"
    assert 2_000_000 <= r[1] < 200_000_000, r[1]
    assert r[2] == 1, "the second role did not leave its wait"
    assert r[3] < 500_000_000, "the second role waited for its own limit instead of the abort flag"
    # read once: the latched timeout; read again: cleared
    assert aqd.device_status() == TIMEOUT
    assert aqd.device_status() == 0


def test_context_usable_after_the_latched_timeout():
    out = torch.zeros(5, dtype=torch.int64, device="cuda")
    aqd.selftest_wait_timeout(out)
    assert aqd.device_status() == TIMEOUT
    wl = synth.config0()
    cv = wl.convs[0]
    xt = oracle.CodeTensor.from_codes(wl.inputs[0], 2)
    W, wp = weights(cv.w, 2)
    want = oracle.conv_int(xt, wp, 2, 0, 3, 3, 1, 1, 64, m0=cv.m0, shift=cv.shift, bias=cv.bias, out_bits=2)
    Y = aqd.DTensor.empty(1, 32, 32, 64, 2)
    aqd.conv_int(to_device(xt), W, 1, 1, Y, rq=aqd.RequantParams.from_numpy(cv.m0, cv.shift, cv.bias))
    torch.cuda.synchronize()
    assert np.array_equal(Y.data.cpu().numpy().reshape(want.packed.shape), want.packed)
    assert aqd.device_status() == 0
