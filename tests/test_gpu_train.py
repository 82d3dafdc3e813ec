"""GPU parity of the training-side steps (Sec. 3.1.2's quantizers with learnable intervals,
Eq. 2 and Eq. 3, their Straight-Through-Estimator backward, and Sec. 3.2.2's per-level batch
statistics) against the oracle (``oracle.train``).

Codes and fake-quantized values are compared bit for bit (both sides decide every code in
float32 in the equations' order). The input gradient is compared exactly; the interval's
gradient is a sum over the tensor, formed in float32 within runs of a thread and in float64
beyond on the GPU (float64 throughout in the oracle), so it is compared within
1e-5 x sum(|gy|) (|dy/dnu| <= 1 for both quantizers, so that bounds 1e-5 x sum(|gy dy/dnu|)
from above). Batch statistics come from float32 runs of 32 shifted values: the mean is compared
within 1e-6 x (|mean| + standard deviation), the variance within 1e-5 relative."""
import numpy as np
import pytest
import torch

from oracle import train as ot
from paper_2007_06919_gb300 import aqd

pytestmark = pytest.mark.gpu


def _cuda(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


@pytest.mark.parametrize("weight", [False, True])
@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_fake_quant_matches_oracle(weight, bits):
    rng = np.random.default_rng(bits * 10 + weight)
    n = 1_000_003  # vector path plus a 3-element tail
    nu = 1.7 if weight else 2.3
    x = (rng.normal(0.0 if weight else 1.0, 1.4, size=n)).astype(np.float32)
    x[:6] = [0.0, nu, -nu, nu * 1.0000001, -1e30, 1e30]
    want_y, want_c = (ot.fake_quant_weight if weight else ot.fake_quant_act)(x, nu, bits)
    y, c = aqd.fake_quant(_cuda(x), nu, bits, weight=weight)
    torch.cuda.synchronize()
    assert np.array_equal(c.cpu().numpy(), want_c)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), want_y.view(np.uint32))
    # a view at a 4-byte offset: the scalar path
    xs = _cuda(x)[1:]
    want_y, want_c = (ot.fake_quant_weight if weight else ot.fake_quant_act)(x[1:], nu, bits)
    y2 = torch.empty(n, dtype=torch.float32, device="cuda")[1:]
    y2, c2 = aqd.fake_quant(xs, nu, bits, weight=weight, y=y2)
    torch.cuda.synchronize()
    assert np.array_equal(c2.cpu().numpy(), want_c)
    assert np.array_equal(y2.cpu().numpy().view(np.uint32), want_y.view(np.uint32))


def _gnu_scale(gy):
    """sum(|gy|): an upper bound of sum(|gy * dy/dnu|), since |dy/dnu| <= 1."""
    return float(np.sum(np.abs(gy.astype(np.float64))))


@pytest.mark.parametrize("weight", [False, True])
@pytest.mark.parametrize("bits", [2, 4, 8])
@pytest.mark.parametrize("n", [0, 1, 37, 2_000_001])
def test_fake_quant_backward_matches_oracle(weight, bits, n):
    rng = np.random.default_rng(n + bits + 5 * weight)
    nu = 0.9 if weight else 1.9
    x = rng.normal(0.0 if weight else 0.8, 1.1, size=n).astype(np.float32)
    gy = rng.normal(0, 1, size=n).astype(np.float32)
    want_gx, want_gnu = (ot.fake_quant_weight_backward if weight else ot.fake_quant_act_backward)(x, gy, nu, bits)
    gx, gnu = aqd.fake_quant_backward(_cuda(x), _cuda(gy), nu, bits, weight=weight)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    assert np.array_equal(gx.cpu().numpy().view(np.uint32), want_gx.view(np.uint32))
    got = float(gnu.cpu().item())
    if n == 0:
        assert got == 0.0
    else:
        assert abs(got - want_gnu) <= 1e-5 * _gnu_scale(gy) + 1e-30


def test_fake_quant_full_size_and_repeatable():
    """A 16x100x168x256 activation tensor (69M values): codes and values bit for bit, and the
    interval's gradient the same on a second run (fixed reduction order)."""
    rng = np.random.default_rng(99)
    x = rng.normal(1.2, 1.0, size=16 * 100 * 168 * 256).astype(np.float32)
    gy = rng.normal(0, 1e-3, size=x.size).astype(np.float32)
    want_y, want_c = ot.fake_quant_act(x, 2.5, 4)
    xd, gd = _cuda(x), _cuda(gy)
    y, c = aqd.fake_quant(xd, 2.5, 4)
    _, g1 = aqd.fake_quant_backward(xd, gd, 2.5, 4)
    _, g2 = aqd.fake_quant_backward(xd, gd, 2.5, 4)
    torch.cuda.synchronize()
    assert np.array_equal(c.cpu().numpy(), want_c)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), want_y.view(np.uint32))
    assert float(g1.item()) == float(g2.item())
    _, want_gnu = ot.fake_quant_act_backward(x, gy, 2.5, 4)
    assert abs(float(g1.item()) - want_gnu) <= 1e-5 * _gnu_scale(gy)


@pytest.mark.parametrize("batch,c", [(2, 256), (1, 96), (3, 7)])
def test_bn_level_stats_matches_oracle(batch, c):
    rng = np.random.default_rng(batch * 1000 + c)
    levels = [(100, 168), (50, 84), (25, 42), (13, 21), (7, 11)]
    zs = []
    for l, (h, w) in enumerate(levels):
        mu = rng.normal(0, 5, size=c)
        sd = rng.uniform(0.1, 3, size=c)
        zs.append((mu + sd * rng.normal(size=(batch, h, w, c))).astype(np.float32))
    zs[4][...] = 3.25  # a constant level: variance exactly 0 on both sides
    want_m, want_v = ot.bn_level_stats(zs)
    m, v = aqd.bn_level_stats([_cuda(z) for z in zs])
    torch.cuda.synchronize()
    m, v = m.cpu().numpy(), v.cpu().numpy()
    assert np.all(np.abs(m - want_m) <= 1e-6 * (np.abs(want_m) + np.sqrt(want_v)) + 1e-12)
    assert np.all(np.abs(v - want_v) <= 1e-5 * want_v + 1e-12)
    assert np.all(v[4] == 0) and np.all(m[4] == 3.25)


def test_training_argument_errors():
    x = torch.zeros(16, dtype=torch.float32, device="cuda")
    for bad in (dict(nu=0.0, bits=2), dict(nu=float("inf"), bits=2), dict(nu=1.0, bits=9), dict(nu=1.0, bits=0)):
        with pytest.raises(aqd.AqdError) as e:
            aqd.fake_quant(x, bad["nu"], bad["bits"])
        assert e.value.status == 1
    with pytest.raises(aqd.AqdError) as e:
        aqd.fake_quant_backward(x, x, -1.0, 2)
    assert e.value.status == 1
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
