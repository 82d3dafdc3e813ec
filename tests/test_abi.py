"""CPU-only checks of the C ABI: libaqd.so loads, exports every entry point that
include/aqd.h declares, and its host-side logic (row sizes, Eq. 8's multiplier search,
argument validation that returns before any launch) is right. No kernel runs here."""
import ctypes
import math
import os
import re
from fractions import Fraction

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2007_06919_gb300 import aqd, build
    build.build()
    return aqd.load()


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "aqd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(aqd_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_abi():
    names = _declared_functions()
    for n in ("aqd_conv_int", "aqd_residual_add_int", "aqd_requant", "aqd_conv_int_grouped",
              "aqd_quantize_multiplier", "aqd_device_status", "aqd_maxpool_codes"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in _declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_library_is_built_for_sm103a():
    from paper_2007_06919_gb300 import build
    assert "arch=compute_103a,code=sm_103a" in " ".join(build.ARCH)


def test_row_bytes_matches_oracle(lib, oracle_mod):
    from paper_2007_06919_gb300 import aqd
    for c in (3, 32, 64, 80, 96, 256, 512):
        for bits in (2, 3, 4, 8, 32):
            assert aqd.row_bytes(c, bits) == oracle_mod.row_bytes(c, bits), (c, bits)


def test_quantize_multiplier_matches_oracle(lib, oracle_mod):
    from paper_2007_06919_gb300 import aqd
    rng = np.random.default_rng(0)
    vals = list(rng.uniform(1e-9, 1.0, 200)) + list(rng.uniform(1, 1e6, 50)) + [0.0, -0.25, 2 ** -40, 0.5]
    for r in vals:
        assert aqd.quantize_multiplier(r) == oracle_mod.quantize_multiplier(r), r
    with pytest.raises(aqd.AqdError):
        aqd.quantize_multiplier(float(2 ** 40))
    with pytest.raises(aqd.AqdError):
        aqd.quantize_multiplier(math.inf)


def test_quantize_multiplier_error_bound(lib):
    """|real - m0 2^-(31+shift)| <= 2^-(32+shift) (half an LSB of the chosen grid)."""
    from paper_2007_06919_gb300 import aqd
    for r in (0.1, 0.7, 3.3, 1e-5):
        m0, sh = aqd.quantize_multiplier(r)
        assert abs(Fraction(r) - Fraction(m0, 2 ** (31 + sh))) <= Fraction(1, 2 ** (32 + sh))


def test_status_strings(lib):
    assert lib.aqd_status_string(0) == b"ok"
    assert lib.aqd_status_string(1) == b"invalid argument"
    assert lib.aqd_status_string(4) == b"device wait timed out"


def test_invalid_arguments_return_before_launch(lib):
    from paper_2007_06919_gb300 import aqd
    # NULL tensors / bad sizes are rejected on the host; nothing reaches the GPU
    assert lib.aqd_conv_int(None, None, 1, 1, 0, None, None, None, None, None, 0, None) == 1
    assert lib.aqd_pack_codes(None, 10, 48, 2, None, None) == 1  # 48 channels at 2 bits
    assert lib.aqd_pack_codes(None, 10, 64, 5, None, None) == 1  # 5-bit codes do not exist
    x = aqd._Tensor(1, 4, 4, 64, 2, 16)
    y = aqd._Tensor(1, 4, 4, 64, 32, 16)  # int32 output: no requant tables needed
    w = aqd._Weights(256, 64, 3, 3, 32, 2, 0)  # cin 32 != x.c 64
    st = lib.aqd_conv_int(ctypes.byref(x), ctypes.byref(w), 1, 1, 0, None, None, None, ctypes.byref(y), None, 0, None)
    assert st == 1
    assert b"cin" in lib.aqd_last_error()
    x2 = aqd._Tensor(1, 4, 4, 64, 2, 8)  # misaligned data pointer
    w2 = aqd._Weights(256, 64, 3, 3, 64, 2, 0)
    st = lib.aqd_conv_int(ctypes.byref(x2), ctypes.byref(w2), 1, 1, 0, None, None, None, ctypes.byref(y), None, 0, None)
    assert st == 1 and b"aligned" in lib.aqd_last_error()
    assert lib.aqd_conv_weights_bytes(0, 3, 3, 64) == 0
    assert lib.aqd_conv_weights_bytes(256, 3, 3, 256) >= 256 * 2304 * 3
    # the split workspace calls check their job list and workspace before anything else
    assert lib.aqd_conv_expand_input(None, 0, ctypes.byref(w2), 1, 1, None, 0, None) == 1
    jobs = (aqd._Job * 1)()
    jobs[0].x = aqd._Tensor(1, 4, 4, 256, 2, 256)
    assert lib.aqd_conv_expand_input(jobs, 1, ctypes.byref(w2), 1, 1, None, 0, None) == 1
    assert b"workspace" in lib.aqd_last_error()
    assert lib.aqd_conv_int_grouped_expanded(jobs, 9, ctypes.byref(w2), 1, 1, None, None, None, 0, None) == 1


def test_workspace_bytes_host_logic(lib):
    """The expanded-activation workspace is planes * sum(n * (h+2p) * (w+2p)) * cin bytes for
    stride-1 convolutions with cin % 128 == 0, or cin % 64 == 0 for codes and weights of at
    most 4 bits (planes = 2 for 8-bit activation codes; 8-bit
    two's-complement weights take the split form), else 0; 8-bit operands also need
    K * 3825 < 2^24 (the exact FP32 partial sums)."""
    from paper_2007_06919_gb300 import aqd
    jobs = (aqd._Job * 2)()
    jobs[0].x = aqd._Tensor(2, 10, 17, 256, 2, 256)
    jobs[1].x = aqd._Tensor(2, 5, 9, 256, 2, 256)
    w = aqd._Weights(256, 256, 3, 3, 256, 2, 0)
    want = (2 * 12 * 19 + 2 * 7 * 11) * 256
    assert lib.aqd_conv_workspace_bytes(jobs, 2, ctypes.byref(w), 1, 1) == want
    assert lib.aqd_conv_workspace_bytes(jobs, 2, ctypes.byref(w), 2, 1) == 0      # stride 2
    w8 = aqd._Weights(256, 256, 3, 3, 256, 8, 0)
    assert lib.aqd_conv_workspace_bytes(jobs, 2, ctypes.byref(w8), 1, 1) == want  # 8-bit weights: split
    w8odd = aqd._Weights(256, 256, 3, 3, 256, 8, 1)
    assert lib.aqd_conv_workspace_bytes(jobs, 2, ctypes.byref(w8odd), 1, 1) == 0  # odd grid, 8-bit
    jobs8 = (aqd._Job * 2)()
    jobs8[0].x = aqd._Tensor(2, 10, 17, 256, 8, 256)
    jobs8[1].x = aqd._Tensor(2, 5, 9, 256, 8, 256)
    assert lib.aqd_conv_workspace_bytes(jobs8, 2, ctypes.byref(w8), 1, 1) == 2 * want  # two planes
    wbig = aqd._Weights(256, 256, 3, 3, 2048, 8, 0)  # K = 18432: 18432 * 3825 >= 2^24
    jobs8[0].x = aqd._Tensor(2, 10, 17, 2048, 8, 256)
    assert lib.aqd_conv_workspace_bytes(jobs8, 1, ctypes.byref(wbig), 1, 1) == 0
    w64 = aqd._Weights(256, 64, 3, 3, 64, 2, 0)
    jobs[0].x = aqd._Tensor(2, 10, 17, 64, 2, 256)
    assert lib.aqd_conv_workspace_bytes(jobs, 1, ctypes.byref(w64), 1, 1) == 2 * 12 * 19 * 64  # 64-byte rows
    w96 = aqd._Weights(256, 96, 3, 3, 96, 2, 0)
    jobs[0].x = aqd._Tensor(2, 10, 17, 96, 2, 256)
    assert lib.aqd_conv_workspace_bytes(jobs, 1, ctypes.byref(w96), 1, 1) == 0    # cin 96
    w64s = aqd._Weights(256, 64, 3, 3, 64, 8, 0)                                   # split weights
    jobs[0].x = aqd._Tensor(2, 10, 17, 64, 2, 256)
    assert lib.aqd_conv_workspace_bytes(jobs, 1, ctypes.byref(w64s), 1, 1) == 0
    jobs[0].x = aqd._Tensor(2, 10, 17, 64, 8, 256)                                # 8-bit codes, cin 64
    assert lib.aqd_conv_workspace_bytes(jobs, 1, ctypes.byref(w64), 1, 1) == 0


def test_set_conv_path_rejects_unknown(lib):
    assert lib.aqd_set_conv_path(7) == -1
    assert lib.aqd_set_conv_path(0) in (0, 1, 2)


def test_training_entry_points_validate_before_any_launch(lib):
    """The training-side entries refuse bad arguments on the host (AQD_ERR_INVALID = 1, no
    CUDA call made); the workspace queries are pure host arithmetic."""
    f32 = ctypes.c_float
    assert lib.aqd_fake_quant_backward_workspace_bytes() >= 8 * 512
    assert lib.aqd_bn_level_stats_workspace_bytes(0, 256) == 0
    assert lib.aqd_bn_level_stats_workspace_bytes(9, 256) == 0
    assert lib.aqd_bn_level_stats_workspace_bytes(5, 0) == 0
    assert lib.aqd_bn_level_stats_workspace_bytes(5, 256) > 0
    fake = ctypes.c_void_p(0x1000)  # never dereferenced: the calls fail before any launch
    for nu, bits, weight in ((0.0, 2, 0), (-1.0, 2, 0), (float("nan"), 2, 0), (float("inf"), 4, 1),
                             (1.0, 0, 0), (1.0, 9, 0), (1.0, 4, 2)):
        assert lib.aqd_fake_quant(fake, 16, f32(nu), bits, weight, fake, None, None) == 1
        assert lib.aqd_fake_quant_backward(fake, fake, 16, f32(nu), bits, weight, fake, fake, fake, 8192, None) == 1
    assert lib.aqd_fake_quant(fake, -1, f32(1.0), 2, 0, fake, None, None) == 1
    assert lib.aqd_fake_quant(fake, 16, f32(1.0), 2, 0, None, None, None) == 1          # no output
    assert lib.aqd_fake_quant(ctypes.c_void_p(0x1002), 16, f32(1.0), 2, 0, fake, None, None) == 1  # misaligned
    assert lib.aqd_fake_quant_backward(fake, fake, 16, f32(1.0), 2, 0, fake, None, fake, 8192, None) == 1  # no gnu
    assert lib.aqd_fake_quant_backward(fake, fake, 16, f32(1.0), 2, 0, fake, fake, fake, 8, None) == 1  # small ws
    ptrs = (ctypes.c_void_p * 1)(fake)
    pix = (ctypes.c_int64 * 1)(10)
    assert lib.aqd_bn_level_stats(ptrs, pix, 0, 4, fake, fake, fake, 1 << 20, None) == 1   # levels
    assert lib.aqd_bn_level_stats(ptrs, pix, 1, 0, fake, fake, fake, 1 << 20, None) == 1   # channels
    assert lib.aqd_bn_level_stats(ptrs, pix, 1, 4, fake, fake, fake, 8, None) == 1         # workspace
    neg = (ctypes.c_int64 * 1)(-1)
    assert lib.aqd_bn_level_stats(ptrs, neg, 1, 4, fake, fake, fake, 1 << 20, None) == 1   # pixels
