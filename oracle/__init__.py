"""CPU oracle for AQD's integer-only quantized convolution (arXiv 2007.06919).

TEST INFRASTRUCTURE, NOT PRODUCT CODE. Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package. It shares no code with the
CUDA path (``paper_2007_06919_gb300``) and never imports it.

The arithmetic lives in ``aqd_ref.c`` (plain C, exact int64); this module only builds
that file into ``liboracle_aqd.so`` and marshals numpy arrays into it with ctypes.

Sections followed: Eq. 2 (Sec. 3.1.2), Eq. 3-4 (Sec. 3.2.1), Eq. 5-6 (Sec. 3.2.2),
Eq. 7-8 (Sec. 3.2.3), Sec. 3.2.4 (max-pooling on codes).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "aqd_ref.c")
_LIB_PATH = os.path.join(_HERE, "liboracle_aqd.so")

W_TWOS = 0
W_ODD = 1


def build(force: bool = False) -> str:
    """Compile aqd_ref.c with gcc (OpenMP over output pixels; results do not depend on it)."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "aqd_ref.h"))
    ):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-Wall", "-Wno-unknown-pragmas",
           _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Tensor(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("h", ctypes.c_int32), ("w", ctypes.c_int32),
                ("c", ctypes.c_int32), ("bits", ctypes.c_int32), ("data", ctypes.c_void_p)]


class _Requant(ctypes.Structure):
    _fields_ = [("m0", ctypes.c_void_p), ("shift", ctypes.c_void_p), ("bias", ctypes.c_void_p),
                ("levels", ctypes.c_int32)]


class _Residual(ctypes.Structure):
    _fields_ = [("skip", ctypes.POINTER(_Tensor)), ("c", ctypes.c_void_p), ("d", ctypes.c_void_p),
                ("upsample", ctypes.c_int32), ("scale_main", ctypes.c_int32)]


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        _lib.aqd_ref_row_bytes.restype = ctypes.c_int64
        _lib.aqd_ref_row_bytes.argtypes = [ctypes.c_int32, ctypes.c_int32]
        _lib.aqd_ref_quantize_multiplier.argtypes = [
            ctypes.c_double, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_int8)]
        _lib.aqd_ref_pack.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                                      ctypes.c_int32, ctypes.c_void_p]
        _lib.aqd_ref_unpack.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                                        ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p]
        i32, i64, vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p
        T, R, S = ctypes.POINTER(_Tensor), ctypes.POINTER(_Requant), ctypes.POINTER(_Residual)
        _lib.aqd_ref_conv_int.argtypes = [T, vp, i32, i32, i32, i32, i32, i32, i32, i32, R, S, i32, T]
        _lib.aqd_ref_conv_int_pixels.argtypes = [T, vp, i32, i32, i32, i32, i32, i32, i32, i32, R, S, i32,
                                                 i32, i32, vp, i64, vp]
        _lib.aqd_ref_requant_tensor.argtypes = [T, R, i32, i32, T]
        _lib.aqd_ref_residual_add_int.argtypes = [T, T, vp, vp, i32, i32, R, i32, i32, T]
        _lib.aqd_ref_maxpool_codes.argtypes = [T, i32, i32, i32, T]
        for fn in ("aqd_ref_pack", "aqd_ref_unpack", "aqd_ref_quantize_multiplier", "aqd_ref_conv_int",
                   "aqd_ref_conv_int_pixels", "aqd_ref_requant_tensor", "aqd_ref_residual_add_int",
                   "aqd_ref_maxpool_codes"):
            getattr(_lib, fn).restype = ctypes.c_int
    return _lib


def _ptr(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


class OracleError(RuntimeError):
    pass


def _check(st: int, what: str):
    if st != 0:
        raise OracleError(f"{what}: oracle returned status {st}")


def row_bytes(c: int, bits: int) -> int:
    return int(lib().aqd_ref_row_bytes(c, bits))


def pack(codes: np.ndarray, bits: int) -> np.ndarray:
    """codes [..., C] int -> packed uint8 [..., row_bytes] (low k bits of each code)."""
    codes = np.ascontiguousarray(codes, dtype=np.int32)
    c = codes.shape[-1]
    rows = codes.size // c
    rb = row_bytes(c, bits)
    if rb < 0:
        raise OracleError(f"no packed layout for C={c} bits={bits}")
    out = np.zeros(codes.shape[:-1] + (rb,), dtype=np.uint8)
    _check(lib().aqd_ref_pack(_ptr(codes), rows, c, bits, _ptr(out)), "pack")
    return out


def unpack(packed: np.ndarray, c: int, bits: int, signed: bool = False) -> np.ndarray:
    """packed uint8 [..., row_bytes] -> codes int32 [..., C] (two's complement if signed)."""
    packed = np.ascontiguousarray(packed, dtype=np.uint8)
    rb = row_bytes(c, bits)
    if rb < 0 or packed.shape[-1] != rb:
        raise OracleError(f"packed rows of {packed.shape[-1]} bytes do not match C={c} bits={bits}")
    rows = packed.size // rb
    out = np.zeros(packed.shape[:-1] + (c,), dtype=np.int32)
    _check(lib().aqd_ref_unpack(_ptr(packed), rows, c, bits, int(signed), _ptr(out)), "unpack")
    return out


def quantize_multiplier(real: float) -> tuple[int, int]:
    m0 = ctypes.c_int32()
    sh = ctypes.c_int8()
    _check(lib().aqd_ref_quantize_multiplier(float(real), ctypes.byref(m0), ctypes.byref(sh)),
           "quantize_multiplier")
    return int(m0.value), int(sh.value)


def _tensor(packed: np.ndarray, n: int, h: int, w: int, c: int, bits: int) -> _Tensor:
    assert packed.flags["C_CONTIGUOUS"]
    rb = row_bytes(c, bits)
    assert packed.nbytes == n * h * w * rb, (packed.nbytes, n, h, w, rb)
    return _Tensor(n, h, w, c, bits, packed.ctypes.data)


def _requant(m0, shift, bias, levels):
    keep = [np.ascontiguousarray(m0, np.int32) if m0 is not None else None,
            np.ascontiguousarray(shift, np.int8) if shift is not None else None,
            np.ascontiguousarray(bias, np.int32) if bias is not None else None]
    return _Requant(_ptr(keep[0]), _ptr(keep[1]), _ptr(keep[2]), levels), keep


class CodeTensor:
    """A packed NHWC tensor as the oracle sees it (bytes + logical shape)."""

    def __init__(self, packed: np.ndarray, n: int, h: int, w: int, c: int, bits: int):
        self.packed = np.ascontiguousarray(packed)
        self.n, self.h, self.w, self.c, self.bits = n, h, w, c, bits

    @classmethod
    def from_codes(cls, codes: np.ndarray, bits: int) -> "CodeTensor":
        n, h, w, c = codes.shape
        if bits == 32:
            return cls(np.ascontiguousarray(codes, np.int32).view(np.uint8).reshape(n, h, w, 4 * c),
                       n, h, w, c, 32)
        return cls(pack(codes, bits), n, h, w, c, bits)

    def codes(self, signed: bool | None = None) -> np.ndarray:
        if self.bits == 32:
            return self.packed.view(np.int32).reshape(self.n, self.h, self.w, self.c).copy()
        return unpack(self.packed, self.c, self.bits, bool(signed)).reshape(self.n, self.h, self.w, self.c)

    def ct(self) -> _Tensor:
        return _tensor(self.packed, self.n, self.h, self.w, self.c, self.bits)


def conv_out_hw(h, w, kh, kw, stride, pad):
    return (h + 2 * pad - kh) // stride + 1, (w + 2 * pad - kw) // stride + 1


def conv_int(x: CodeTensor, w_packed: np.ndarray, w_bits: int, w_format: int, kh: int, kw: int,
             stride: int, pad: int, cout: int, *, level: int = 0, m0=None, shift=None, bias=None,
             levels: int = 1, skip: CodeTensor | None = None, skip_c=None, skip_d=None,
             upsample: int = 1, scale_main: int = 0, out_bits: int = 2) -> CodeTensor:
    """Full oracle convolution (Eq. 4 -> Eq. 6 -> Eq. 7 -> Eq. 2); returns packed output."""
    ho, wo = conv_out_hw(x.h, x.w, kh, kw, stride, pad)
    rb = row_bytes(cout, out_bits)
    if rb < 0 or ho <= 0 or wo <= 0:
        raise OracleError("bad output geometry")
    y = np.zeros((x.n, ho, wo, rb), dtype=np.uint8)
    yt = _tensor(y, x.n, ho, wo, cout, out_bits)
    rq, keep = _requant(m0, shift, bias, levels)
    rqp = ctypes.byref(rq) if (m0 is not None or bias is not None or out_bits != 32) else None
    if out_bits == 32 and m0 is None and bias is None:
        rqp = None
    res = None
    keep2 = []
    if skip is not None:
        st = skip.ct()
        keep2 = [st, np.ascontiguousarray(skip_c, np.int32), np.ascontiguousarray(skip_d, np.int8)]
        res = _Residual(ctypes.pointer(st), _ptr(keep2[1]), _ptr(keep2[2]), upsample, scale_main)
    w_packed = np.ascontiguousarray(w_packed, np.uint8)
    _check(lib().aqd_ref_conv_int(ctypes.byref(x.ct()), _ptr(w_packed), w_bits, w_format, kh, kw,
                                  stride, pad, cout, level, rqp,
                                  ctypes.byref(res) if res is not None else None, out_bits,
                                  ctypes.byref(yt)), "conv_int")
    return CodeTensor(y, x.n, ho, wo, cout, out_bits)


def conv_int_pixels(x: CodeTensor, w_packed: np.ndarray, w_bits: int, w_format: int, kh: int,
                    kw: int, stride: int, pad: int, cout: int, pix: np.ndarray, *, level: int = 0,
                    m0=None, shift=None, bias=None, levels: int = 1,
                    skip: CodeTensor | None = None, skip_c=None, skip_d=None, upsample: int = 1,
                    scale_main: int = 0, out_bits: int = 2) -> np.ndarray:
    """Oracle outputs (unpacked int32 [len(pix), cout]) for selected flattened output pixels."""
    ho, wo = conv_out_hw(x.h, x.w, kh, kw, stride, pad)
    pix = np.ascontiguousarray(pix, np.int64)
    out = np.zeros((pix.size, cout), dtype=np.int32)
    rq, keep = _requant(m0, shift, bias, levels)
    rqp = ctypes.byref(rq)
    if out_bits == 32 and m0 is None and bias is None:
        rqp = None
    res = None
    keep2 = []
    if skip is not None:
        st = skip.ct()
        keep2 = [st, np.ascontiguousarray(skip_c, np.int32), np.ascontiguousarray(skip_d, np.int8)]
        res = _Residual(ctypes.pointer(st), _ptr(keep2[1]), _ptr(keep2[2]), upsample, scale_main)
    w_packed = np.ascontiguousarray(w_packed, np.uint8)
    _check(lib().aqd_ref_conv_int_pixels(ctypes.byref(x.ct()), _ptr(w_packed), w_bits, w_format,
                                         kh, kw, stride, pad, cout, level, rqp,
                                         ctypes.byref(res) if res is not None else None, out_bits,
                                         ho, wo, _ptr(pix), pix.size, _ptr(out)), "conv_int_pixels")
    return out


def requant(acc: CodeTensor, m0, shift, bias, *, level: int = 0, levels: int = 1,
            out_bits: int = 2) -> CodeTensor:
    rb = row_bytes(acc.c, out_bits)
    y = np.zeros((acc.n, acc.h, acc.w, rb), dtype=np.uint8)
    yt = _tensor(y, acc.n, acc.h, acc.w, acc.c, out_bits)
    rq, keep = _requant(m0, shift, bias, levels)
    _check(lib().aqd_ref_requant_tensor(ctypes.byref(acc.ct()), ctypes.byref(rq), level, out_bits,
                                        ctypes.byref(yt)), "requant")
    return CodeTensor(y, acc.n, acc.h, acc.w, acc.c, out_bits)


def residual_add(a: CodeTensor, b: CodeTensor, c, d, *, upsample: int = 1, scale_a: int = 0,
                 m0=None, shift=None, bias=None, level: int = 0, levels: int = 1,
                 out_bits: int = 2) -> CodeTensor:
    rb = row_bytes(a.c, out_bits)
    y = np.zeros((a.n, a.h, a.w, rb), dtype=np.uint8)
    yt = _tensor(y, a.n, a.h, a.w, a.c, out_bits)
    c = np.ascontiguousarray(c, np.int32)
    d = np.ascontiguousarray(d, np.int8)
    rqp = None
    keep = None
    if m0 is not None or bias is not None:
        rq, keep = _requant(m0, shift, bias, levels)
        rqp = ctypes.byref(rq)
    _check(lib().aqd_ref_residual_add_int(ctypes.byref(a.ct()), ctypes.byref(b.ct()), _ptr(c), _ptr(d),
                                          upsample, scale_a, rqp, level, out_bits, ctypes.byref(yt)),
           "residual_add")
    return CodeTensor(y, a.n, a.h, a.w, a.c, out_bits)


def maxpool(x: CodeTensor, k: int, stride: int, pad: int) -> CodeTensor:
    ho, wo = conv_out_hw(x.h, x.w, k, k, stride, pad)
    y = np.zeros((x.n, ho, wo, row_bytes(x.c, x.bits)), dtype=np.uint8)
    yt = _tensor(y, x.n, ho, wo, x.c, x.bits)
    _check(lib().aqd_ref_maxpool_codes(ctypes.byref(x.ct()), k, stride, pad, ctypes.byref(yt)), "maxpool")
    return CodeTensor(y, x.n, ho, wo, x.c, x.bits)


def run_network(layers, tensors: dict) -> dict:
    """Runs a layer list (convs and max-pools naming their input, output and skip tensors)
    on the oracle, in list order. ``tensors`` maps names to CodeTensors and receives every
    layer output. A conv with several jobs (the shared head) takes parameter row l for job l
    (multi-level BN, Sec. 3.2.2); each job is one plain oracle convolution (Eq. 4 -> Eq. 6 ->
    Eq. 7 -> Eq. 2); a max-pool compares codes (Sec. 3.2.4)."""
    for ly in layers:
        if ly.pool is not None:
            k, s, p = ly.pool
            tensors[ly.dst[0]] = maxpool(tensors[ly.src[0]], k, s, p)
            continue
        cv = ly.conv
        wp = pack(cv.w.reshape(-1, cv.cin), cv.w_bits)
        ref = cv.m0 if cv.m0 is not None else cv.bias
        levels = ref.shape[0]
        for j, (src, dst) in enumerate(zip(ly.src, ly.dst)):
            skip = tensors[ly.skip[j]] if ly.skip else None
            tensors[dst] = conv_int(tensors[src], wp, cv.w_bits, W_TWOS, cv.kh, cv.kw, cv.stride, cv.pad,
                                    cv.cout, level=j, m0=cv.m0, shift=cv.shift, bias=cv.bias, levels=levels,
                                    skip=skip, skip_c=cv.skip_c, skip_d=cv.skip_d, upsample=ly.upsample,
                                    out_bits=cv.out_bits)
    return tensors
