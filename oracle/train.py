"""CPU oracle for the training-side steps of AQD (arXiv 2007.06919): the quantizers of Eq. 2
(activations) and Eq. 3 (weights) with learnable intervals (Sec. 3.1.2), their backward pass
under the Straight-Through Estimator, and the per-level batch statistics of the multi-level
batch normalization (Sec. 3.2.2).

TEST INFRASTRUCTURE, NOT PRODUCT CODE: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import it. It shares no code with the CUDA path.

Plain numpy, element by element as the equations read. Each integer code is decided in
float32, the precision the kernels use (``x / nu`` as one correctly rounded float32
division, the clip, the scale by Q = 2^b - 1, then floor(v + 0.5)), so that both sides take
the same rounding decisions; every sum is taken in float64.
"""
from __future__ import annotations

import numpy as np

f32 = np.float32


def _q(bits: int) -> np.float32:
    return f32((1 << bits) - 1)


def fake_quant_act(x: np.ndarray, nu: float, bits: int):
    """Eq. 2: eta = round(clip(x / nu, 0, 1) * (2^b - 1)), x_bar = eta * nu / (2^b - 1).
    Returns (x_bar float32, eta uint8). "round" is half-up (floor(v + 0.5))."""
    x = np.asarray(x, dtype=f32)
    q = _q(bits)
    v = np.clip(x / f32(nu), f32(0), f32(1)) * q
    eta = np.floor(v + f32(0.5))
    s = f32(nu) / q                     # the magnitude-restore scale nu / (2^b - 1)
    return (eta * s).astype(f32), eta.astype(np.uint8)


def fake_quant_weight(w: np.ndarray, nu: float, bits: int):
    """Eq. 3: eta = round((clip(w / nu, -1, 1) + 1) / 2 * (2^b - 1)),
    w_bar = (eta * 2 / (2^b - 1) - 1) * nu. Returns (w_bar float32, eta uint8)."""
    w = np.asarray(w, dtype=f32)
    q = _q(bits)
    v = (np.clip(w / f32(nu), f32(-1), f32(1)) + f32(1)) * f32(0.5) * q
    eta = np.floor(v + f32(0.5))
    wbar = (eta * f32(2) / q - f32(1)) * f32(nu)
    return wbar.astype(f32), eta.astype(np.uint8)


def fake_quant_act_backward(x: np.ndarray, gy: np.ndarray, nu: float, bits: int):
    """The STE backward of Eq. 2 (the rounding's derivative taken as 1):
    d x_bar / d x = 1 for 0 < x / nu < 1, else 0;
    d x_bar / d nu = eta / Q - x / nu inside, 1 where x / nu >= 1, 0 where x / nu <= 0.
    Returns (gx float32, gnu float64 = sum of gy * d x_bar / d nu)."""
    x = np.asarray(x, dtype=f32)
    gy = np.asarray(gy, dtype=f32)
    q = _q(bits)
    v = x / f32(nu)
    inside = (v > 0) & (v < 1)
    eta = np.floor(np.clip(v, f32(0), f32(1)) * q + f32(0.5))
    dnu = np.where(inside, eta / q - v, np.where(v >= 1, f32(1), f32(0))).astype(f32)
    gx = np.where(inside, gy, f32(0)).astype(f32)
    gnu = float(np.sum(gy.astype(np.float64) * dnu.astype(np.float64)))
    return gx, gnu


def fake_quant_weight_backward(w: np.ndarray, gy: np.ndarray, nu: float, bits: int):
    """The STE backward of Eq. 3: d w_bar / d w = 1 for -1 < w / nu < 1, else 0;
    d w_bar / d nu = 2 eta / Q - 1 - w / nu inside, 1 where w / nu >= 1, -1 where w / nu <= -1.
    Returns (gw float32, gnu float64)."""
    w = np.asarray(w, dtype=f32)
    gy = np.asarray(gy, dtype=f32)
    q = _q(bits)
    v = w / f32(nu)
    inside = (v > -1) & (v < 1)
    eta = np.floor((np.clip(v, f32(-1), f32(1)) + f32(1)) * f32(0.5) * q + f32(0.5))
    dnu = np.where(inside, eta * f32(2) / q - f32(1) - v, np.where(v >= 1, f32(1), f32(-1))).astype(f32)
    gw = np.where(inside, gy, f32(0)).astype(f32)
    gnu = float(np.sum(gy.astype(np.float64) * dnu.astype(np.float64)))
    return gw, gnu


def bn_level_stats(levels):
    """Sec. 3.2.2's multi-level BN during training: for each FPN level's tensor z_l (any
    leading shape, channels last), the per-channel batch mean and biased variance over all of
    its pixels, in float64. Returns (mean [L, C], var [L, C])."""
    means, vars_ = [], []
    for z in levels:
        zz = np.asarray(z, dtype=np.float64).reshape(-1, np.shape(z)[-1])
        m = zz.mean(axis=0)
        means.append(m)
        vars_.append(((zz - m) ** 2).mean(axis=0))
    return np.stack(means), np.stack(vars_)
