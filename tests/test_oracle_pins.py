"""Pins of the CPU oracle against what the paper and plain mathematics fix.

None of these compare the oracle with itself: each expected value comes from a hand-worked
example (tests/golden), a textbook routine (numpy int64 matmul, a real-valued convolution),
the paper's float formulas before their integer rewrite (tests/fakequant.py), brute force
over Eq. 8's search space, or an invariant. A dropped term, a wrong sign, a transposed
operand or a wrong tap order in the oracle fails at least one of them.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import fakequant as fq
from paper_2007_06919_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_lines(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]


def _pack_w(oracle, w, bits):
    """weights [cout, kh, kw, cin] signed ints -> packed rows (two's complement fields)."""
    return oracle.pack(w.reshape(-1, w.shape[-1]), bits)


# ------------------------------------------------------------------ packed layout


def test_layout_golden(oracle_mod):
    for ln in _golden_lines("layout.txt"):
        lhs, rhs = ln.split("->")
        bits, c, spec = lhs.split()
        bits, c = int(bits), int(c)
        codes = np.zeros((1, c), np.int32)
        if spec == "ramp4":
            codes[0] = np.arange(c) % 4
        else:
            for kv in spec.split(","):
                i, v = kv.split(":")
                codes[0, int(i)] = int(v)
        want = bytes(int(b, 16) for b in rhs.split())
        got = oracle_mod.pack(codes, bits).tobytes()
        assert got == want, (ln, got.hex())
        assert (oracle_mod.unpack(np.frombuffer(want, np.uint8)[None], c, bits) == codes).all()


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_pack_roundtrip_signed_and_unsigned(oracle_mod, bits):
    rng = np.random.default_rng(7)
    c = 96
    u = rng.integers(0, 1 << bits, size=(5, c)).astype(np.int32)
    assert (oracle_mod.unpack(oracle_mod.pack(u, bits), c, bits) == u).all()
    s = rng.integers(-(1 << (bits - 1)), 1 << (bits - 1), size=(5, c)).astype(np.int32)
    assert (oracle_mod.unpack(oracle_mod.pack(s, bits), c, bits, signed=True) == s).all()


def test_row_bytes(oracle_mod):
    assert oracle_mod.row_bytes(256, 2) == 64
    assert oracle_mod.row_bytes(256, 3) == 96
    assert oracle_mod.row_bytes(256, 4) == 128
    assert oracle_mod.row_bytes(3, 8) == 3
    assert oracle_mod.row_bytes(80, 32) == 320
    assert oracle_mod.row_bytes(48, 2) == -1  # 2/3/4-bit rows need C % 32 == 0


# ------------------------------------------------------------------ hand-worked examples


def test_hand_1x1(oracle_mod):
    x = np.zeros((1, 1, 1, 32), np.int32)
    x[0, 0, 0, :2] = (3, 2)
    # 32 identical output channels (k-bit output rows hold 32 codes at a time)
    w = np.zeros((32, 1, 1, 32), np.int32)
    w[:, 0, 0, :2] = (1, -1)
    xt = oracle_mod.CodeTensor.from_codes(x, 2)
    wp = _pack_w(oracle_mod, w, 2)
    full = lambda v: np.full((1, 32), v, np.int64)  # noqa: E731
    for ln in _golden_lines("hand_1x1.txt"):
        lhs, rhs = ln.split("->")
        f = lhs.split()
        shift, bias = int(f[0]), int(f[1])
        out_bits = int(f[5])
        mirror = len(f) > 6 and f[6] == "mirror"
        kw = dict(m0=full(1 << 30), shift=full(shift), bias=full(bias), out_bits=out_bits)
        if f[2] != "none":
            s = np.full((1, 1, 1, 32), int(f[2]), np.int32)
            kw.update(skip=oracle_mod.CodeTensor.from_codes(s, 32), skip_c=full(int(f[3])),
                      skip_d=full(int(f[4])), scale_main=int(mirror))
        y = oracle_mod.conv_int(xt, wp, 2, oracle_mod.W_TWOS, 1, 1, 1, 0, 32, **kw)
        assert (y.codes()[0, 0, 0, :] == int(rhs)).all(), ln


def _grid(s):
    return np.array([[int(v) for v in row.split()] for row in s.split("/")])


def test_hand_3x3(oracle_mod):
    g = {}
    for ln in _golden_lines("hand_3x3.txt"):
        k, v = ln.split("=")
        g[k.strip()] = _grid(v)
    x = np.zeros((1, 3, 3, 32), np.int32)
    x[..., 0] = 1
    w = np.zeros((32, 3, 3, 32), np.int32)
    w[..., 0] = 1
    xt = oracle_mod.CodeTensor.from_codes(x, 2)
    wp = _pack_w(oracle_mod, w, 2)
    z = np.zeros((1, 32))
    y = oracle_mod.conv_int(xt, wp, 2, 0, 3, 3, 1, 1, 32, bias=z, out_bits=32).codes()
    assert (y[0] == g["s1_int32"][:, :, None]).all()
    y = oracle_mod.conv_int(xt, wp, 2, 0, 3, 3, 1, 1, 32, m0=np.full((1, 32), 1 << 30),
                            shift=np.ones((1, 32)), bias=z, out_bits=2).codes()
    assert (y[0] == g["s1_2bit"][:, :, None]).all()
    y = oracle_mod.conv_int(xt, wp, 2, 0, 3, 3, 2, 1, 32, bias=z, out_bits=32).codes()
    assert (y[0] == g["s2_int32"][:, :, None]).all()


# ------------------------------------------------------------------ structure: one-hot


def test_one_hot_activation_reproduces_weight_slice(oracle_mod):
    """A single code 1 at input (h0, w0, c0) makes output (h0-r+1, w0-s+1, n) equal
    w[n, r, s, c0] (stride 1, pad 1, int32 output, bias 0): pins tap order and layout."""
    rng = np.random.default_rng(3)
    h0, w0, c0 = 2, 3, 37
    x = np.zeros((1, 5, 6, 64), np.int32)
    x[0, h0, w0, c0] = 1
    w = rng.integers(-1, 2, size=(8, 3, 3, 64)).astype(np.int32)
    y = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, 2), _pack_w(oracle_mod, w, 2), 2, 0,
                            3, 3, 1, 1, 8, bias=np.zeros((1, 8)), out_bits=32).codes()
    want = np.zeros((1, 5, 6, 8), np.int64)
    for r in range(3):
        for s in range(3):
            want[0, h0 - r + 1, w0 - s + 1, :] = w[:, r, s, c0]
    assert (y == want).all()


def test_one_hot_weight_shifts_input(oracle_mod):
    """A weight that is 1 only at tap (r, s) of channel c reads input channel c shifted by
    (r - 1, s - 1): y[h, w] = x[h + r - 1, w + s - 1, c] (zero outside)."""
    rng = np.random.default_rng(4)
    x = rng.integers(0, 16, size=(2, 6, 7, 32)).astype(np.int32)
    for (r, s, c) in [(0, 0, 5), (2, 1, 31), (1, 2, 0)]:
        w = np.zeros((1, 3, 3, 32), np.int32)
        w[0, r, s, c] = 1
        y = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, 4), _pack_w(oracle_mod, w, 4), 4, 0,
                                3, 3, 1, 1, 1, bias=np.zeros((1, 1)), out_bits=32).codes()[..., 0]
        xp = np.pad(x[..., c], ((0, 0), (1, 1), (1, 1)))
        assert (y == xp[:, r:r + 6, s:s + 7]).all()


# ------------------------------------------------------------------ textbook routines


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_1x1_equals_numpy_int64_matmul(oracle_mod, bits):
    rng = np.random.default_rng(10 + bits)
    x = synth.act_codes(rng, (2, 3, 5, 64), bits)
    w = synth.weight_codes(rng, (48, 1, 1, 64), bits)
    y = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, bits), _pack_w(oracle_mod, w, bits),
                            bits, 0, 1, 1, 1, 0, 48, bias=np.zeros((1, 48)), out_bits=32).codes()
    want = x.reshape(-1, 64).astype(np.int64) @ w.reshape(48, 64).T.astype(np.int64)
    assert (y.reshape(-1, 48) == want).all()


@pytest.mark.parametrize("k,stride,pad", [(3, 1, 1), (3, 2, 1), (1, 2, 0), (7, 2, 3), (3, 1, 0)])
def test_conv_equals_real_convolution(oracle_mod, k, stride, pad):
    rng = np.random.default_rng(k * 10 + stride)
    x = synth.act_codes(rng, (2, 9, 11, 32), 4)
    w = synth.weight_codes(rng, (16, k, k, 32), 4)
    y = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, 4), _pack_w(oracle_mod, w, 4), 4, 0,
                            k, k, stride, pad, 16, bias=np.zeros((1, 16)), out_bits=32).codes()
    want = fq.conv2d_real(x, w, stride, pad)  # exact: small integers in float64
    assert (y == want).all()


def test_odd_weight_format_is_eq4_identity(oracle_mod):
    """Eq. 4: sum x_bar * w_bar over real values equals eta_conv * alpha_conv with
    eta_conv = sum eta_x (2 eta_w - 2^b + 1) and alpha_conv = nu_x nu_w / (2^b - 1)^2."""
    rng = np.random.default_rng(5)
    b = 3
    nu_x, nu_w = 1.7, 0.45
    x_real = rng.uniform(-0.3, 2.2, size=(1, 6, 6, 32))
    w_real = rng.normal(0, 0.3, size=(8, 3, 3, 32))
    eta_x = fq.quantize_act(x_real, nu_x, b).astype(np.int32)
    eta_w = fq.quantize_weight(w_real, nu_w, b).astype(np.int32)
    real = fq.conv2d_real(fq.dequant_act(eta_x, nu_x, b), fq.dequant_weight_odd(eta_w, nu_w, b), 1, 1)
    wp = oracle_mod.pack(eta_w.reshape(-1, 32), b)
    eta_conv = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(eta_x, b), wp, b, oracle_mod.W_ODD,
                                   3, 3, 1, 1, 8, bias=np.zeros((1, 8)), out_bits=32).codes()
    alpha_conv = nu_x * nu_w / ((1 << b) - 1) ** 2
    np.testing.assert_allclose(eta_conv * alpha_conv, real, rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------------ invariants


def test_all_zero_codes_map_to_clip_bias(oracle_mod):
    rng = np.random.default_rng(6)
    cout = 64
    m0, shift, bias = synth.requant_params(rng, 1, cout, shift_lo=0, shift_hi=4, bias_lim=40)
    x = np.zeros((1, 4, 4, 32), np.int32)
    w = synth.weight_codes(rng, (cout, 3, 3, 32), 2)
    y = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, 2), _pack_w(oracle_mod, w, 2), 2, 0,
                            3, 3, 1, 1, cout, m0=m0, shift=shift, bias=bias, out_bits=4).codes()
    for n in range(cout):
        v = Fraction(int(bias[0, n]) * int(m0[0, n]), 2 ** (31 + int(shift[0, n])))
        want = min(max(math.floor(v + Fraction(1, 2)), 0), 15)
        assert (y[..., n] == want).all()


def test_unit_multiplier_gives_clip_acc_plus_bias(oracle_mod):
    """M0 = 2^30 with shift = -1 is the multiplier 2^30 / 2^30 = 1 exactly."""
    rng = np.random.default_rng(8)
    x = synth.act_codes(rng, (1, 5, 5, 32), 2)
    w = synth.weight_codes(rng, (32, 3, 3, 32), 2)
    bias = rng.integers(-5, 6, size=(1, 32)).astype(np.int32)
    args = (oracle_mod.CodeTensor.from_codes(x, 2), _pack_w(oracle_mod, w, 2), 2, 0, 3, 3, 1, 1, 32)
    y = oracle_mod.conv_int(*args, m0=np.full((1, 32), 1 << 30), shift=np.full((1, 32), -1),
                            bias=bias, out_bits=3).codes()
    acc = fq.conv2d_real(x, w, 1, 1)
    assert (y == np.clip(acc + bias[0], 0, 7)).all()


def test_outputs_in_code_range_and_monotone_in_bias(oracle_mod):
    wl = synth.config0()
    cv = wl.convs[0]
    xt = oracle_mod.CodeTensor.from_codes(wl.inputs[0], 2)
    wp = _pack_w(oracle_mod, cv.w, 2)
    prev = None
    for delta in (-300, 0, 300):
        y = oracle_mod.conv_int(xt, wp, 2, 0, 3, 3, 1, 1, 64, m0=cv.m0, shift=np.full_like(cv.shift, 2),
                                bias=cv.bias + delta, out_bits=2).codes()
        assert y.min() >= 0 and y.max() <= 3
        if prev is not None:
            assert (y >= prev).all()
        prev = y


# ------------------------------------------------------------------ Eq. 7 special cases


def test_skip_unit_ratio_is_plain_add(oracle_mod):
    """alpha_1 = alpha_2 gives F = 1 (c = 2^d): the skip is an integer add."""
    rng = np.random.default_rng(9)
    a = rng.integers(-1000, 1000, size=(1, 3, 4, 32)).astype(np.int32)
    b = rng.integers(0, 16, size=(1, 3, 4, 32)).astype(np.int32)
    for d in (0, 5, 30):
        y = oracle_mod.residual_add(oracle_mod.CodeTensor.from_codes(a, 32), oracle_mod.CodeTensor.from_codes(b, 4),
                                    np.full((1, 32), 1 << d), np.full((1, 32), d), out_bits=32).codes()
        assert (y == a + b).all()


def test_skip_power_of_two_is_fqn_shift(oracle_mod):
    """Eq. 9 (FQN) is Eq. 8 with c = 1: the skip contributes round(eta_s / 2^d)."""
    rng = np.random.default_rng(11)
    a = rng.integers(-1000, 1000, size=(1, 2, 5, 32)).astype(np.int32)
    b = rng.integers(-5000, 5000, size=(1, 2, 5, 32)).astype(np.int32)
    for d in (1, 3, 7):
        y = oracle_mod.residual_add(oracle_mod.CodeTensor.from_codes(a, 32), oracle_mod.CodeTensor.from_codes(b, 32),
                                    np.ones((1, 32)), np.full((1, 32), d), out_bits=32).codes()
        assert (y == a + np.floor(b / 2 ** d + 0.5).astype(np.int64)).all()


def test_residual_add_matches_conv_epilogue(oracle_mod):
    """residual_add(a, b) equals the conv epilogue with a as the accumulator: a 1x1 conv
    with an identity weight reproduces a, so both paths must agree bit for bit."""
    rng = np.random.default_rng(12)
    x = synth.act_codes(rng, (2, 4, 6, 32), 4)
    skip = synth.act_codes(rng, (2, 2, 3, 32), 4)
    w = np.zeros((32, 1, 1, 32), np.int32)
    w[np.arange(32), 0, 0, np.arange(32)] = 1
    m0, shift, bias = synth.requant_params(rng, 1, 32, shift_lo=-2, shift_hi=1, bias_lim=3)
    c, d = synth.skip_params(rng, 1, 32, np.full((1, 32), 28))
    for mirror in (0, 1):
        y1 = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, 4), _pack_w(oracle_mod, w, 4), 4, 0,
                                 1, 1, 1, 0, 32, m0=m0, shift=shift, bias=bias,
                                 skip=oracle_mod.CodeTensor.from_codes(skip, 4), skip_c=c, skip_d=d,
                                 upsample=2, scale_main=mirror, out_bits=4).codes()
        y2 = oracle_mod.residual_add(oracle_mod.CodeTensor.from_codes(x, 4), oracle_mod.CodeTensor.from_codes(skip, 4),
                                     c, d, upsample=2, scale_a=mirror, m0=m0, shift=shift, bias=bias,
                                     out_bits=4).codes()
        assert (y1 == y2).all()


# ------------------------------------------------------------------ Eq. 8: F(m, n)


def _best_error(r: Fraction):
    best = None
    for d in range(0, 63):
        c = math.floor(abs(r) * 2 ** d + Fraction(1, 2))
        if c >= 2 ** 31:
            continue
        err = abs(abs(r) - Fraction(c, 2 ** d))
        best = err if best is None or err < best else best
    return best


def test_quantize_multiplier_is_eq8_argmin(oracle_mod):
    rng = np.random.default_rng(13)
    vals = list(rng.uniform(1e-6, 1.0, 40)) + list(rng.uniform(1.0, 3e4, 20)) + [0.5, 1 / 3, 2 ** -20, 0.999999999]
    for r in vals:
        m0, sh = oracle_mod.quantize_multiplier(r)
        got = Fraction(m0, 2 ** (31 + sh))
        assert abs(Fraction(r) - got) == _best_error(Fraction(r)), r
        assert 0 <= 31 + sh <= 62 and 0 < m0 < 2 ** 31
    assert oracle_mod.quantize_multiplier(-0.3) == (-oracle_mod.quantize_multiplier(0.3)[0],
                                                    oracle_mod.quantize_multiplier(0.3)[1])
    assert oracle_mod.quantize_multiplier(0.0) == (0, 0)


# ------------------------------------------------------------------ paper's float formulas


def _bn_setup(rng, cout):
    gamma = rng.uniform(0.5, 1.5, cout) * rng.choice([-1, 1], cout, p=[0.2, 0.8])
    beta = rng.normal(0, 0.5, cout)
    mu = rng.normal(0, 0.5, cout)
    var = rng.uniform(0.5, 2.0, cout)
    return gamma, beta, mu, var


def test_exact_dyadic_fake_quant(oracle_mod):
    """With dyadic scales every float64 step is exact, so Eq. 4-7 applied to real values
    (BN as multiply-add, real skip add, Eq. 2 quantizer with round-half-up) must equal the
    oracle's integer codes exactly."""
    rng = np.random.default_rng(14)
    b, cin, cout = 4, 32, 32
    x = synth.act_codes(rng, (2, 6, 7, cin), b)
    w = synth.weight_codes(rng, (cout, 3, 3, cin), b)
    skip = synth.act_codes(rng, (2, 6, 7, cout), b)
    alpha_x, alpha_w = 2.0 ** -3, 2.0 ** -5            # dequant steps of x and w
    alpha_conv = alpha_x * alpha_w
    s_int = rng.integers(-60, 60, cout)                  # s of Eq. 5, integer here
    k_mult = rng.integers(1, 16, cout) * 2.0 ** -6       # alpha_z (2^b-1)/nu_next, 4 significant bits
    j = rng.integers(1, 4, cout)                         # alpha_skip / alpha_z = integer j (F exact)
    # nu_next = 2^b - 1 makes Eq. 2's scale (2^b - 1) / nu_next exactly 1, so alpha_z = k_mult
    nu_next = float((1 << b) - 1)
    alpha_z = k_mult * nu_next / ((1 << b) - 1)
    conv_real = fq.conv2d_real(x * alpha_x, w * alpha_w, 1, 1)
    z = (conv_real / alpha_conv + s_int) * alpha_z      # Eq. 5, third line
    y_real = z + skip * (j * alpha_z)                    # Eq. 7 first line, alpha_skip = j alpha_z
    want = fq.quantize_act_exact(y_real, nu_next, b)
    m0 = np.zeros((1, cout), np.int64)
    shift = np.zeros((1, cout), np.int64)
    for n in range(cout):
        m0[0, n], shift[0, n] = oracle_mod.quantize_multiplier(k_mult[n])
        assert Fraction(int(m0[0, n]), 2 ** (31 + int(shift[0, n]))) == Fraction(k_mult[n])
    got = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, b), _pack_w(oracle_mod, w, b), b, 0, 3, 3, 1, 1,
                              cout, m0=m0, shift=shift, bias=s_int[None],
                              skip=oracle_mod.CodeTensor.from_codes(skip, b), skip_c=j[None] * 4,
                              skip_d=np.full((1, cout), 2), out_bits=b).codes()
    assert (got == want).all()
    assert len(np.unique(got)) > 4  # not a degenerate all-clip case


@pytest.mark.parametrize("mirror", [0, 1])
def test_real_bn_fake_quant_within_one_lsb(oracle_mod, mirror):
    """Arbitrary real BN parameters (Eq. 5) folded to bias = round(s), (M0, shift) =
    F(alpha_z (2^b-1) / nu_next) and (c, d) = F(ratio of skip scales) (Eq. 8): the integer
    codes stay within one LSB of Eq. 2 applied to the real-valued BN + skip output."""
    rng = np.random.default_rng(15 + mirror)
    b, cin, cout = 3, 64, 32
    nu_x, nu_w, nu_skip, nu_next = 2.0, 0.8, 3.0, 2.5
    x = synth.act_codes(rng, (1, 8, 9, cin), b)
    w = synth.weight_codes(rng, (cout, 3, 3, cin), b)
    skip = synth.act_codes(rng, (1, 8, 9, cout), b)
    alpha_x = nu_x / ((1 << b) - 1)
    alpha_w = nu_w / 3.0
    alpha_conv = alpha_x * alpha_w
    gamma, beta, mu, var = _bn_setup(rng, cout)
    gamma = np.abs(gamma)  # alpha_z > 0 keeps the skip-direction choice per channel simple
    eps = 1e-5
    sd = np.sqrt(var + eps)
    s = (beta * sd / gamma - mu) / alpha_conv            # Eq. 5
    alpha_z = alpha_conv * gamma / sd
    alpha_s = nu_skip / ((1 << b) - 1)
    z = fq.batch_norm(fq.conv2d_real(x * alpha_x, w * alpha_w, 1, 1), mu, var, eps, gamma, beta)
    y_real = z + skip * alpha_s
    want = fq.quantize_act(y_real, nu_next, b)
    m0 = np.zeros((1, cout), np.int64); sh = np.zeros((1, cout), np.int64)
    c = np.zeros((1, cout), np.int64); d = np.zeros((1, cout), np.int64)
    bias = np.floor(s + 0.5).astype(np.int64)[None]
    for n in range(cout):
        if mirror:
            # main branch expressed in skip units: (eta_conv + s) alpha_z = (..) F(alpha_z/alpha_s) alpha_s
            ratio = alpha_z[n] / alpha_s
            out_scale = alpha_s
        else:
            ratio = alpha_s / alpha_z[n]
            out_scale = alpha_z[n]
        cm, cs = oracle_mod.quantize_multiplier(ratio)
        c[0, n], d[0, n] = cm, 31 + cs
        if d[0, n] > 62 or d[0, n] < 0:
            pytest.skip("ratio outside Eq. 8's shift range")
        m0[0, n], sh[0, n] = oracle_mod.quantize_multiplier(out_scale * ((1 << b) - 1) / nu_next)
    got = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, b), _pack_w(oracle_mod, w, b), b, 0, 3, 3, 1, 1,
                              cout, m0=m0, shift=sh, bias=bias,
                              skip=oracle_mod.CodeTensor.from_codes(skip, b), skip_c=c, skip_d=d,
                              scale_main=mirror, out_bits=b).codes()
    diff = np.abs(got.astype(np.int64) - want.astype(np.int64))
    assert diff.max() <= 1
    assert (diff == 0).mean() > 0.6
    assert len(np.unique(got)) >= 4


def test_round_half_up_not_half_even(oracle_mod):
    """Eq. 2's nearest-integer with ties upward: 2.5 -> 3 and 0.5 -> 1 at the requant."""
    acc = np.array([5, 1, -1, 3], np.int32).reshape(1, 1, 4, 1)
    acc = np.repeat(acc, 32, axis=3)
    y = oracle_mod.requant(oracle_mod.CodeTensor.from_codes(acc, 32), np.full((1, 32), 1 << 30),
                           np.zeros((1, 32)), np.zeros((1, 32)), out_bits=2).codes()
    assert list(y[0, 0, :, 0]) == [3, 1, 0, 2]


def test_requant_saturates_before_multiply(oracle_mod):
    """bias + acc beyond int32 saturates to the int32 limit before the rescale."""
    acc = np.full((1, 1, 1, 32), 2 ** 31 - 10, np.int32)
    y = oracle_mod.requant(oracle_mod.CodeTensor.from_codes(acc, 32), np.full((1, 32), 1 << 30),
                           np.full((1, 32), 31), np.full((1, 32), 100), out_bits=32).codes()
    assert (y == 2 ** 31 - 1).all()


# ------------------------------------------------------------------ Sec. 3.2.4: max-pool


def test_maxpool_commutes_with_dequant(oracle_mod):
    rng = np.random.default_rng(16)
    x = synth.act_codes(rng, (2, 9, 10, 64), 4)
    y = oracle_mod.maxpool(oracle_mod.CodeTensor.from_codes(x, 4), 3, 2, 1).codes()
    alpha = 0.37
    want = fq.maxpool_real(x * alpha, 3, 2, 1)
    np.testing.assert_allclose(y * alpha, want, rtol=0, atol=1e-12)


# ------------------------------------------------------------------ Eq. 7 with Sec. 3.2.4's 2x up-read


def _dyadic_upsample_case(rng, b, cin, cout, n, h, w):
    """Codes and dyadic scales for an exact float64 restatement of Eq. 4 -> Eq. 7 -> Eq. 2 in
    which the skip is the coarser map of the FPN top-down path, read through nearest 2x
    upsampling. h and w are odd and differ, so a swapped or ceil-rounded up-index fails."""
    x = synth.act_codes(rng, (n, h, w, cin), b)
    wt = synth.weight_codes(rng, (cout, 3, 3, cin), b)
    skip = synth.act_codes(rng, (n, (h + 1) // 2, (w + 1) // 2, cout), b)
    s_int = rng.integers(-40, 40, cout)
    k_mult = rng.integers(1, 16, cout) * 2.0 ** -6     # M0 / 2^R, four significant bits
    j = rng.integers(1, 4, cout)                        # integer ratio of the two scales
    return x, wt, skip, s_int, k_mult, j


def _multipliers(oracle_mod, k_mult):
    cout = k_mult.size
    m0 = np.zeros((1, cout), np.int64)
    shift = np.zeros((1, cout), np.int64)
    for i in range(cout):
        m0[0, i], shift[0, i] = oracle_mod.quantize_multiplier(k_mult[i])
        assert Fraction(int(m0[0, i]), 2 ** (31 + int(shift[0, i]))) == Fraction(k_mult[i])
    return m0, shift


def _eq7_real(acc_real, s_int, skip_up, j, k_mult, mirror, b):
    """Eq. 7's real sum quantized by Eq. 2 (nu_next = 2^b - 1, so Eq. 2's scale is 1).
    Default direction: the skip is in units j * alpha_z of the main branch's scale alpha_z.
    Mirror: the main branch is in units j * alpha_s of the skip's scale alpha_s. The
    output multiplier is k_mult per unit of the finer scale in both cases."""
    if mirror:
        y_real = ((acc_real + s_int) * j + skip_up) * k_mult
    else:
        y_real = (acc_real + s_int + skip_up * j) * k_mult
    return fq.quantize_act_exact(y_real, float((1 << b) - 1), b)


@pytest.mark.parametrize("mirror", [0, 1])
def test_conv_upsample2_skip_exact_fake_quant(oracle_mod, mirror):
    """Sec. 3.2.4's FPN top-down add as Eq. 7 inside the conv epilogue: the skip tensor is
    the coarser map, read at (ho // 2, wo // 2) by nearest upsampling. The float64
    restatement upsamples with numpy (repeat along H and W), crops to the output and adds
    in real arithmetic; with dyadic scales each float step is exact, so the oracle's codes
    must match exactly on an odd, non-square output (9 x 13)."""
    rng = np.random.default_rng(40 + mirror)
    b, cin, cout, n, h, w = 4, 32, 32, 2, 9, 13
    x, wt, skip, s_int, k_mult, j = _dyadic_upsample_case(rng, b, cin, cout, n, h, w)
    alpha_x, alpha_w = 2.0 ** -3, 2.0 ** -5
    acc_real = fq.conv2d_real(x * alpha_x, wt * alpha_w, 1, 1) / (alpha_x * alpha_w)
    skip_up = fq.upsample_nearest2(skip)[:, :h, :w, :]
    want = _eq7_real(acc_real, s_int, skip_up, j, k_mult, mirror, b)
    m0, shift = _multipliers(oracle_mod, k_mult)
    got = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, b), _pack_w(oracle_mod, wt, b), b, 0, 3, 3, 1, 1,
                              cout, m0=m0, shift=shift, bias=s_int[None],
                              skip=oracle_mod.CodeTensor.from_codes(skip, b), skip_c=j[None] * 4,
                              skip_d=np.full((1, cout), 2), upsample=2, scale_main=mirror, out_bits=b).codes()
    assert (got == want).all()
    assert len(np.unique(got)) > 4
    # the up-read matters here: the same call without it (skip at full resolution, rows
    # and columns repeated by hand) gives the same codes, and a skip that is not repeated
    # does not
    full = np.ascontiguousarray(skip_up)
    again = oracle_mod.conv_int(oracle_mod.CodeTensor.from_codes(x, b), _pack_w(oracle_mod, wt, b), b, 0, 3, 3, 1, 1,
                                cout, m0=m0, shift=shift, bias=s_int[None],
                                skip=oracle_mod.CodeTensor.from_codes(full, b), skip_c=j[None] * 4,
                                skip_d=np.full((1, cout), 2), upsample=1, scale_main=mirror, out_bits=b).codes()
    assert (again == want).all()


@pytest.mark.parametrize("mirror", [0, 1])
def test_residual_add_upsample2_exact_fake_quant(oracle_mod, mirror):
    """The standalone integer skip add (Eq. 7, then Eq. 2) with the coarser operand read by
    nearest 2x upsampling, against the float64 restatement (numpy repeat, crop, real add)."""
    rng = np.random.default_rng(42 + mirror)
    b, c, n, h, w = 3, 64, 2, 7, 11
    acc = rng.integers(-3000, 3000, size=(n, h, w, c)).astype(np.int32)
    skip = synth.act_codes(rng, (n, (h + 1) // 2, (w + 1) // 2, c), b)
    s_int = rng.integers(-40, 40, c)
    k_mult = rng.integers(1, 16, c) * 2.0 ** -9
    j = rng.integers(1, 4, c)
    want = _eq7_real(acc.astype(np.float64), s_int, fq.upsample_nearest2(skip)[:, :h, :w, :], j, k_mult, mirror, b)
    m0, shift = _multipliers(oracle_mod, k_mult)
    got = oracle_mod.residual_add(oracle_mod.CodeTensor.from_codes(acc, 32), oracle_mod.CodeTensor.from_codes(skip, b),
                                  j[None] * 8, np.full((1, c), 3), upsample=2, scale_a=mirror, m0=m0, shift=shift,
                                  bias=s_int[None], out_bits=b).codes()
    assert (got == want).all()
    assert len(np.unique(got)) > 3


# ------------------------------------------------------------------ the sampled-pixel entry


@pytest.mark.parametrize("stride,upsample", [(1, 2), (2, 1)])
def test_conv_int_pixels_matches_definition(oracle_mod, stride, upsample):
    """conv_int_pixels (the oracle's entry for sampled output pixels, flattened as
    (image, ho, wo) in row-major order) gives, at any list of pixels (unsorted, repeated,
    from every image, at the ragged borders), the codes of the float64 restatement at those
    pixels, and the same rows as the full convolution."""
    rng = np.random.default_rng(44 + stride)
    b, cin, cout, n, h, w = 4, 32, 64, 3, 9, 13
    x, wt, _, s_int, k_mult, j = _dyadic_upsample_case(rng, b, cin, cout, n, h, w)
    ho, wo = (h + 2 - 3) // stride + 1, (w + 2 - 3) // stride + 1
    skip = synth.act_codes(rng, (n, (ho + upsample - 1) // upsample, (wo + upsample - 1) // upsample, cout), b)
    alpha_x, alpha_w = 2.0 ** -3, 2.0 ** -5
    acc_real = fq.conv2d_real(x * alpha_x, wt * alpha_w, stride, 1) / (alpha_x * alpha_w)
    skip_up = (fq.upsample_nearest2(skip) if upsample == 2 else skip)[:, :ho, :wo, :]
    want = _eq7_real(acc_real, s_int, skip_up, j, k_mult, 0, b).reshape(n * ho * wo, cout)
    m0, shift = _multipliers(oracle_mod, k_mult)
    total = n * ho * wo
    corners = [0, wo - 1, (ho - 1) * wo, total - 1, ho * wo, ho * wo + wo - 1, 2 * ho * wo + 3]
    pix = np.concatenate([rng.permutation(total)[:40], corners, corners[:3]])
    rng.shuffle(pix)
    kw = dict(m0=m0, shift=shift, bias=s_int[None], skip=oracle_mod.CodeTensor.from_codes(skip, b),
              skip_c=j[None] * 4, skip_d=np.full((1, cout), 2), upsample=upsample, out_bits=b)
    xt = oracle_mod.CodeTensor.from_codes(x, b)
    wp = _pack_w(oracle_mod, wt, b)
    got = oracle_mod.conv_int_pixels(xt, wp, b, 0, 3, 3, stride, 1, cout, pix, **kw)
    assert got.shape == (pix.size, cout)
    assert (got == want[pix]).all()
    full = oracle_mod.conv_int(xt, wp, b, 0, 3, 3, stride, 1, cout, **kw).codes().reshape(total, cout)
    assert (got == full[pix]).all()
    assert len(np.unique(got)) > 4
