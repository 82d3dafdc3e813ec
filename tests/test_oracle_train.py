"""Pins of the training-side oracle (Eq. 2-3 quantizers with learnable intervals, their STE
backward, the multi-level BN statistics of Sec. 3.2.2) against facts that do not come from
the oracle itself: exact grid values, the quantization error bound, the odd symmetry of Eq. 3,
autograd of a straight-through restatement of the forward, and closed forms of mean and
variance."""
import numpy as np
import pytest
import torch

from oracle import train as ot


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_act_grid_is_exact(bits):
    # nu / Q = 2^-4 exactly, so k * nu / Q are exact float32 values and every grid point
    # maps to its own code and back to itself; out of range clips to 0 / Q
    q = (1 << bits) - 1
    nu = q / 16.0
    k = np.arange(q + 1)
    x = (k / 16.0).astype(np.float32)
    xb, eta = ot.fake_quant_act(x, nu, bits)
    assert np.array_equal(eta, k.astype(np.uint8))
    assert np.array_equal(xb, x)
    xb, eta = ot.fake_quant_act(np.array([-1.0, -1e-6, nu * 2, 1e9], np.float32), nu, bits)
    assert eta.tolist() == [0, 0, q, q]
    assert xb.tolist() == [0.0, 0.0, np.float32(nu), np.float32(nu)]


@pytest.mark.parametrize("bits", [2, 4, 8])
def test_act_error_bound_and_codes(bits):
    rng = np.random.default_rng(bits)
    q = (1 << bits) - 1
    nu = 2.7
    x = rng.normal(1.0, 1.5, size=20000).astype(np.float32)
    xb, eta = ot.fake_quant_act(x, nu, bits)
    ref = np.clip(x.astype(np.float64), 0, nu)
    assert np.max(np.abs(xb - ref)) <= nu / (2 * q) * (1 + 1e-5)
    assert eta.min() == 0 and eta.max() == q
    # x_bar lies on the grid eta * nu / Q
    assert np.allclose(xb, eta.astype(np.float64) * nu / q, rtol=1e-6, atol=0)


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_weight_grid_symmetry_and_bound(bits):
    rng = np.random.default_rng(10 + bits)
    q = (1 << bits) - 1
    nu = 0.8
    w = rng.normal(0.0, 0.6, size=20000).astype(np.float32)
    wb, eta = ot.fake_quant_weight(w, nu, bits)
    wbn, etan = ot.fake_quant_weight(-w, nu, bits)
    # Eq. 3's grid is symmetric: eta(-w) = Q - eta(w) except where (v + 1) / 2 * Q sits at a
    # rounding tie (within float32 rounding of one)
    v = (np.clip(w.astype(np.float64) / nu, -1, 1) + 1) / 2 * q
    far = np.abs(v - np.floor(v) - 0.5) > 1e-4
    assert np.array_equal(etan[far].astype(int), q - eta[far].astype(int))
    assert np.allclose(wbn[far], -wb[far], rtol=0, atol=1e-6)
    # grid values (2 k / Q - 1) nu and the error bound nu / Q
    assert np.allclose(wb, (2 * eta.astype(np.float64) / q - 1) * nu, rtol=1e-6, atol=1e-7)
    assert np.max(np.abs(wb - np.clip(w, -nu, nu))) <= nu / q * (1 + 1e-5)
    assert set(np.unique(eta)) <= set(range(q + 1))


def _ste_autograd(x, gy, nu, bits, weight):
    """Autograd of a float64 restatement of Eq. 2 / Eq. 3 in which the rounding passes the
    gradient straight through (u + (round(u) - u).detach()); returns (gx, gnu)."""
    q = (1 << bits) - 1
    xt = torch.tensor(x, dtype=torch.float64, requires_grad=True)
    nut = torch.tensor(nu, dtype=torch.float64, requires_grad=True)
    if weight:
        u = (torch.clamp(xt / nut, -1, 1) + 1) / 2 * q
        eta = u + (torch.floor(u + 0.5) - u).detach()
        y = (eta * 2 / q - 1) * nut
    else:
        u = torch.clamp(xt / nut, 0, 1) * q
        eta = u + (torch.floor(u + 0.5) - u).detach()
        y = eta * nut / q
    (y * torch.tensor(gy, dtype=torch.float64)).sum().backward()
    return xt.grad.numpy(), float(nut.grad)


@pytest.mark.parametrize("weight", [False, True])
@pytest.mark.parametrize("bits", [2, 4])
def test_ste_backward_matches_autograd(weight, bits):
    rng = np.random.default_rng(bits + 7 * weight)
    nu = 1.3
    x = (rng.normal(0.2, 1.2, size=5000)).astype(np.float32)
    gy = rng.normal(0, 1, size=5000).astype(np.float32)
    # keep away from rounding ties and from the clip boundaries (measure-zero conventions)
    q = (1 << bits) - 1
    v = x.astype(np.float64) / nu
    u = ((np.clip(v, -1, 1) + 1) / 2 if weight else np.clip(v, 0, 1)) * q
    keep = (np.abs(u - np.floor(u) - 0.5) > 1e-3) & (np.abs(np.abs(v) - 1) > 1e-4) & (np.abs(v) > 1e-4)
    x, gy = x[keep], gy[keep]
    f = ot.fake_quant_weight_backward if weight else ot.fake_quant_act_backward
    gx, gnu = f(x, gy, nu, bits)
    ax, anu = _ste_autograd(x, gy, nu, bits, weight)
    # the same zero pattern; inside, the chain rule's (Q / nu) (nu / Q) is 1 to a float64 ulp
    assert np.array_equal(gx == 0, ax == 0)
    assert np.allclose(gx.astype(np.float64), ax, rtol=1e-12, atol=0)
    scale = float(np.sum(np.abs(gy.astype(np.float64))))
    assert abs(gnu - anu) <= 1e-6 * scale


def test_bn_level_stats_closed_forms():
    rng = np.random.default_rng(0)
    c = 7
    # constant level: mean = the constant, variance 0
    z0 = np.full((2, 3, 5, c), 1.25, np.float32)
    # a +-b pattern around a per channel: mean a, variance b^2
    a = rng.normal(0, 3, size=c)
    b = rng.uniform(0.5, 2, size=c)
    sign = np.where(np.arange(40) % 2 == 0, 1.0, -1.0)[:, None]
    z1 = (a + sign * b).astype(np.float64)
    mean, var = ot.bn_level_stats([z0, z1])
    assert np.allclose(mean[0], 1.25) and np.allclose(var[0], 0)
    assert np.allclose(mean[1], a, atol=1e-12) and np.allclose(var[1], b * b, rtol=1e-12)
    # shift and scale: var(k z + s) = k^2 var(z), mean(k z + s) = k mean(z) + s
    z2 = rng.normal(0, 1, size=(3, 11, 13, c))
    m2, v2 = ot.bn_level_stats([z2])
    m3, v3 = ot.bn_level_stats([3.0 * z2 - 5.0])
    assert np.allclose(m3, 3 * m2 - 5) and np.allclose(v3, 9 * v2)
