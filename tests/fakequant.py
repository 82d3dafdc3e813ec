"""Float64 fake-quantized restatement of AQD's layers, used only to pin the oracle.

It works on real values the way the paper defines them before any integer rewrite:
  * activations x_bar = eta_x * nu_x / (2^b - 1)                      (Eq. 2)
  * weights     w_bar = (2 eta_w / (2^b - 1) - 1) nu_w  (odd grid)     (Eq. 3)
                or w_int * alpha_w for a symmetric two's-complement grid
  * conv in real arithmetic on x_bar, w_bar                           (Eq. 4, first line)
  * batch norm z = (conv - mu) / sqrt(var + eps) * gamma + beta        (Eq. 5, first line)
  * skip y = z + x_skip (real sum)                                      (Eq. 7, first line)
  * output code = round(clip(y / nu_next, 0, 1) (2^k - 1))             (Eq. 2 on the next layer)
Nothing here uses the integer rewrite (bias = round(s), M0/shift, c/2^d), so agreement
with the oracle checks that rewrite.
"""
from __future__ import annotations

import numpy as np


def round_half_up(v):
    return np.floor(np.asarray(v, dtype=np.float64) + 0.5)


def quantize_act(x, nu, bits):
    """Eq. 2: codes of real activations x for interval nu."""
    return round_half_up(np.clip(np.asarray(x, np.float64) / nu, 0.0, 1.0) * ((1 << bits) - 1))


def quantize_act_exact(x, nu, bits):
    """Eq. 2 written as round(clip(x * (2^b - 1) / nu, 0, 2^b - 1)), the same function;
    exact in float64 when (2^b - 1) / nu is a power of two and x is dyadic."""
    scale = ((1 << bits) - 1) / nu
    return round_half_up(np.clip(np.asarray(x, np.float64) * scale, 0.0, float((1 << bits) - 1)))


def dequant_act(eta, nu, bits):
    return np.asarray(eta, np.float64) * (nu / ((1 << bits) - 1))


def quantize_weight(w, nu, bits):
    """Eq. 3: eta_w = round((clip(w/nu, -1, 1) + 1) / 2 (2^b - 1))."""
    return round_half_up((np.clip(np.asarray(w, np.float64) / nu, -1.0, 1.0) + 1.0) / 2.0 * ((1 << bits) - 1))


def dequant_weight_odd(eta, nu, bits):
    """Eq. 3 second line: w_bar = (2 eta / (2^b - 1) - 1) nu."""
    return (2.0 * np.asarray(eta, np.float64) / ((1 << bits) - 1) - 1.0) * nu


def conv2d_real(x, w, stride, pad):
    """Direct real-valued convolution, NHWC input and [cout, kh, kw, cin] weights."""
    x = np.asarray(x, np.float64)
    w = np.asarray(w, np.float64)
    n, h, wd, c = x.shape
    cout, kh, kw, cin = w.shape
    assert cin == c
    xp = np.zeros((n, h + 2 * pad, wd + 2 * pad, c), np.float64)
    xp[:, pad:pad + h, pad:pad + wd, :] = x
    ho = (h + 2 * pad - kh) // stride + 1
    wo = (wd + 2 * pad - kw) // stride + 1
    out = np.zeros((n, ho, wo, cout), np.float64)
    for r in range(kh):
        for s in range(kw):
            patch = xp[:, r:r + stride * (ho - 1) + 1:stride, s:s + stride * (wo - 1) + 1:stride, :]
            out += np.tensordot(patch, w[:, r, s, :], axes=([3], [1]))
    return out


def batch_norm(v, mu, var, eps, gamma, beta):
    """Eq. 5 first line, per channel (last axis)."""
    return (v - mu) / np.sqrt(var + eps) * gamma + beta


def upsample_nearest2(v):
    return np.repeat(np.repeat(v, 2, axis=1), 2, axis=2)


def maxpool_real(x, k, stride, pad):
    x = np.asarray(x, np.float64)
    n, h, w, c = x.shape
    xp = np.full((n, h + 2 * pad, w + 2 * pad, c), -np.inf)
    xp[:, pad:pad + h, pad:pad + w, :] = x
    ho = (h + 2 * pad - k) // stride + 1
    wo = (w + 2 * pad - k) // stride + 1
    out = np.full((n, ho, wo, c), -np.inf)
    for r in range(k):
        for s in range(k):
            out = np.maximum(out, xp[:, r:r + stride * (ho - 1) + 1:stride, s:s + stride * (wo - 1) + 1:stride, :])
    return out
