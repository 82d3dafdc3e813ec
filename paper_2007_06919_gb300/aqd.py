"""Thin ctypes binding of libaqd (include/aqd.h), with the same entry-point names.

Only argument marshalling happens here: every step of the integer convolution path runs
in libaqd's CUDA kernels. PyTorch supplies device memory and the current stream. There is
no CPU fallback: if the library or a GPU is missing the calls raise.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

from . import build as _build

W_TWOS = 0
W_ODD = 1

STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported", 3: "CUDA error", 4: "device wait timed out",
          5: "device check failed"}


class AqdError(RuntimeError):
    def __init__(self, status: int, func: str, msg: str):
        super().__init__(f"{func}: {STATUS.get(status, status)}: {msg}")
        self.status = status


class _Tensor(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int32), ("h", ctypes.c_int32), ("w", ctypes.c_int32), ("c", ctypes.c_int32),
                ("bits", ctypes.c_int32), ("data", ctypes.c_void_p)]


class _Requant(ctypes.Structure):
    _fields_ = [("m0", ctypes.c_void_p), ("shift", ctypes.c_void_p), ("bias", ctypes.c_void_p),
                ("levels", ctypes.c_int32)]


class _Skip(ctypes.Structure):
    _fields_ = [("c", ctypes.c_void_p), ("d", ctypes.c_void_p), ("upsample", ctypes.c_int32),
                ("scale_main", ctypes.c_int32)]


class _Weights(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("cout", ctypes.c_int32), ("kh", ctypes.c_int32),
                ("kw", ctypes.c_int32), ("cin", ctypes.c_int32), ("w_bits", ctypes.c_int32),
                ("w_format", ctypes.c_int32)]


class _Job(ctypes.Structure):
    _fields_ = [("x", _Tensor), ("y", _Tensor), ("skip", _Tensor), ("level", ctypes.c_int32)]


EXPORTS = ["aqd_row_bytes", "aqd_quantize_multiplier", "aqd_status_string", "aqd_last_error",
           "aqd_device_status", "aqd_set_conv_path", "aqd_last_conv_path", "aqd_pack_codes",
           "aqd_unpack_codes", "aqd_conv_weights_bytes", "aqd_conv_prepare_weights", "aqd_conv_int",
           "aqd_conv_int_grouped", "aqd_conv_workspace_bytes", "aqd_conv_expand_input",
           "aqd_conv_int_grouped_expanded", "aqd_conv_int_grouped_chain", "aqd_requant", "aqd_residual_add_int",
           "aqd_maxpool_codes", "aqd_maxpool_expand", "aqd_conv_int_static_workspace", "aqd_selftest_wait_timeout",
           "aqd_conv_tower_sync_bytes", "aqd_conv_int_grouped_tower", "aqd_fake_quant",
           "aqd_fake_quant_backward_workspace_bytes", "aqd_fake_quant_backward",
           "aqd_bn_level_stats_workspace_bytes", "aqd_bn_level_stats"]

_lib = None


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Loads libaqd.so (building it in-tree first if it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise FileNotFoundError(f"{path} is not built")
        _build.build()
    L = ctypes.CDLL(path)
    c_int, i32, i64, vp = ctypes.c_int, ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p
    L.aqd_row_bytes.restype = i64
    L.aqd_row_bytes.argtypes = [i32, i32]
    L.aqd_quantize_multiplier.argtypes = [ctypes.c_double, ctypes.POINTER(i32), ctypes.POINTER(ctypes.c_int8)]
    L.aqd_status_string.restype = ctypes.c_char_p
    L.aqd_status_string.argtypes = [c_int]
    L.aqd_last_error.restype = ctypes.c_char_p
    L.aqd_device_status.argtypes = [vp, ctypes.POINTER(i32)]
    L.aqd_set_conv_path.restype = i32
    L.aqd_set_conv_path.argtypes = [i32]
    L.aqd_last_conv_path.restype = i32
    L.aqd_pack_codes.argtypes = [vp, i64, i32, i32, vp, vp]
    L.aqd_unpack_codes.argtypes = [vp, i64, i32, i32, i32, vp, vp]
    L.aqd_conv_weights_bytes.restype = ctypes.c_size_t
    L.aqd_conv_weights_bytes.argtypes = [i32, i32, i32, i32]
    L.aqd_conv_prepare_weights.argtypes = [vp, ctypes.POINTER(_Weights), vp, ctypes.c_size_t, vp]
    L.aqd_conv_int.argtypes = [ctypes.POINTER(_Tensor), ctypes.POINTER(_Weights), i32, i32, i32,
                               ctypes.POINTER(_Requant), ctypes.POINTER(_Tensor), ctypes.POINTER(_Skip),
                               ctypes.POINTER(_Tensor), vp, ctypes.c_size_t, vp]
    L.aqd_conv_int_grouped.argtypes = [ctypes.POINTER(_Job), i32, ctypes.POINTER(_Weights), i32, i32,
                                       ctypes.POINTER(_Requant), ctypes.POINTER(_Skip), vp, ctypes.c_size_t, vp]
    L.aqd_conv_expand_input.argtypes = [ctypes.POINTER(_Job), i32, ctypes.POINTER(_Weights), i32, i32, vp,
                                        ctypes.c_size_t, vp]
    L.aqd_conv_int_grouped_expanded.argtypes = L.aqd_conv_int_grouped.argtypes
    L.aqd_conv_int_grouped_chain.argtypes = [ctypes.POINTER(_Job), i32, ctypes.POINTER(_Weights), i32, i32,
                                             ctypes.POINTER(_Requant), ctypes.POINTER(_Skip), vp, ctypes.c_size_t,
                                             i32, vp, ctypes.c_size_t, vp]
    L.aqd_conv_int_static_workspace.argtypes = [ctypes.POINTER(_Tensor), ctypes.POINTER(_Weights), i32, i32, i32,
                                                ctypes.POINTER(_Requant), ctypes.POINTER(_Tensor),
                                                ctypes.POINTER(_Skip), ctypes.POINTER(_Tensor), vp]
    L.aqd_conv_int_static_workspace.restype = c_int
    L.aqd_conv_tower_sync_bytes.restype = ctypes.c_size_t
    L.aqd_conv_tower_sync_bytes.argtypes = [ctypes.POINTER(_Job), i32, i32, i32]
    L.aqd_conv_int_grouped_tower.argtypes = [ctypes.POINTER(_Job), i32, i32, ctypes.POINTER(_Weights),
                                             ctypes.POINTER(_Requant), i32, vp, vp, ctypes.c_size_t, vp,
                                             ctypes.c_size_t, i32, vp]
    L.aqd_conv_int_grouped_tower.restype = c_int
    L.aqd_selftest_wait_timeout.argtypes = [vp, vp]
    L.aqd_selftest_wait_timeout.restype = c_int
    L.aqd_conv_workspace_bytes.restype = ctypes.c_size_t
    L.aqd_conv_workspace_bytes.argtypes = [ctypes.POINTER(_Job), i32, ctypes.POINTER(_Weights), i32, i32]
    L.aqd_requant.argtypes = [ctypes.POINTER(_Tensor), ctypes.POINTER(_Requant), i32, ctypes.POINTER(_Tensor), vp]
    L.aqd_residual_add_int.argtypes = [ctypes.POINTER(_Tensor), ctypes.POINTER(_Tensor), ctypes.POINTER(_Skip),
                                       ctypes.POINTER(_Requant), i32, ctypes.POINTER(_Tensor), vp]
    L.aqd_maxpool_codes.argtypes = [ctypes.POINTER(_Tensor), i32, i32, i32, ctypes.POINTER(_Tensor), vp]
    L.aqd_maxpool_expand.argtypes = [ctypes.POINTER(_Tensor), i32, i32, i32, ctypes.POINTER(_Tensor),
                                     ctypes.POINTER(_Weights), i32, i32, vp, ctypes.c_size_t, vp]
    f32, i64, sz = ctypes.c_float, ctypes.c_int64, ctypes.c_size_t
    L.aqd_fake_quant.argtypes = [vp, i64, f32, i32, i32, vp, vp, vp]
    L.aqd_fake_quant_backward_workspace_bytes.restype = sz
    L.aqd_fake_quant_backward_workspace_bytes.argtypes = []
    L.aqd_fake_quant_backward.argtypes = [vp, vp, i64, f32, i32, i32, vp, vp, vp, sz, vp]
    L.aqd_bn_level_stats_workspace_bytes.restype = sz
    L.aqd_bn_level_stats_workspace_bytes.argtypes = [i32, i32]
    L.aqd_bn_level_stats.argtypes = [ctypes.POINTER(vp), ctypes.POINTER(i64), i32, i32, vp, vp, vp, sz, vp]
    for name in ("aqd_quantize_multiplier", "aqd_device_status", "aqd_pack_codes", "aqd_unpack_codes",
                 "aqd_conv_prepare_weights", "aqd_conv_int", "aqd_conv_int_grouped", "aqd_conv_expand_input",
                 "aqd_conv_int_grouped_expanded", "aqd_conv_int_grouped_chain", "aqd_requant",
                 "aqd_residual_add_int", "aqd_maxpool_codes", "aqd_maxpool_expand", "aqd_fake_quant",
                 "aqd_fake_quant_backward", "aqd_bn_level_stats"):
        getattr(L, name).restype = c_int
    _lib = L
    return L


def _check(st: int, func: str):
    if st != 0:
        msg = load().aqd_last_error().decode(errors="replace")
        raise AqdError(st, func, msg)


def _stream(stream=None) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _ptr(t: torch.Tensor | None):
    if t is None:
        return None
    assert t.is_cuda and t.is_contiguous(), "device tensors must be contiguous CUDA tensors"
    return t.data_ptr()


# ------------------------------------------------------------------ tensors


def row_bytes(c: int, bits: int) -> int:
    return int(load().aqd_row_bytes(c, bits))


@dataclass
class DTensor:
    """A packed NHWC code tensor (or int32 tensor) in device memory."""
    data: torch.Tensor  # uint8 [n, h, w, row_bytes] (any contiguous byte buffer of that size)
    n: int
    h: int
    w: int
    c: int
    bits: int

    @classmethod
    def empty(cls, n, h, w, c, bits, device="cuda"):
        rb = row_bytes(c, bits)
        if rb < 0:
            raise ValueError(f"no packed layout for C={c} at {bits} bits")
        return cls(torch.empty((n, h, w, rb), dtype=torch.uint8, device=device), n, h, w, c, bits)

    @classmethod
    def from_codes(cls, codes: torch.Tensor, bits: int) -> "DTensor":
        """codes: int32 CUDA tensor [n, h, w, c]."""
        n, h, w, c = codes.shape
        if bits == 32:
            data = codes.to(torch.int32).contiguous().view(torch.uint8).reshape(n, h, w, 4 * c)
            return cls(data, n, h, w, c, 32)
        out = cls.empty(n, h, w, c, bits, device=codes.device)
        pack_codes(codes.reshape(-1, c), bits, out=out.data)
        return out

    def codes(self, signed: bool = False) -> torch.Tensor:
        if self.bits == 32:
            return self.data.contiguous().view(torch.int32).reshape(self.n, self.h, self.w, self.c)
        return unpack_codes(self.data.reshape(-1, row_bytes(self.c, self.bits)), self.c, self.bits,
                            signed).reshape(self.n, self.h, self.w, self.c)

    def ct(self) -> _Tensor:
        assert self.data.numel() * self.data.element_size() == self.n * self.h * self.w * row_bytes(self.c, self.bits)
        return _Tensor(self.n, self.h, self.w, self.c, self.bits, _ptr(self.data))


def pack_codes(codes: torch.Tensor, bits: int, out: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """codes: int32 CUDA [rows, c] -> packed uint8 [rows, row_bytes]."""
    codes = codes.to(torch.int32).contiguous()
    c = codes.shape[-1]
    rows = codes.numel() // c
    rb = row_bytes(c, bits)
    if out is None:
        out = torch.empty((rows, rb), dtype=torch.uint8, device=codes.device)
    _check(load().aqd_pack_codes(_ptr(codes), rows, c, bits, _ptr(out), _stream(stream)), "aqd_pack_codes")
    return out


def unpack_codes(packed: torch.Tensor, c: int, bits: int, signed: bool = False, stream=None) -> torch.Tensor:
    packed = packed.contiguous()
    rb = row_bytes(c, bits)
    rows = packed.numel() // rb
    out = torch.empty((rows, c), dtype=torch.int32, device=packed.device)
    _check(load().aqd_unpack_codes(_ptr(packed), rows, c, bits, int(signed), _ptr(out), _stream(stream)),
           "aqd_unpack_codes")
    return out


# ------------------------------------------------------------------ parameters


@dataclass
class RequantParams:
    m0: torch.Tensor | None      # int32 [levels, cout]
    shift: torch.Tensor | None   # int8  [levels, cout]
    bias: torch.Tensor | None    # int32 [levels, cout]
    levels: int

    @classmethod
    def from_numpy(cls, m0, shift, bias, device="cuda"):
        def t(a, dt):
            return None if a is None else torch.as_tensor(a).to(dt).contiguous().to(device)
        ref = m0 if m0 is not None else bias
        return cls(t(m0, torch.int32), t(shift, torch.int8), t(bias, torch.int32), int(ref.shape[0]))

    def c(self) -> _Requant:
        return _Requant(_ptr(self.m0), _ptr(self.shift), _ptr(self.bias), self.levels)


@dataclass
class SkipParams:
    c: torch.Tensor     # int32 [levels, cout]
    d: torch.Tensor     # int8  [levels, cout]
    upsample: int = 1
    scale_main: int = 0

    @classmethod
    def from_numpy(cls, c, d, upsample=1, scale_main=0, device="cuda"):
        return cls(torch.as_tensor(c).to(torch.int32).contiguous().to(device),
                   torch.as_tensor(d).to(torch.int8).contiguous().to(device), upsample, scale_main)

    def cs(self) -> _Skip:
        return _Skip(_ptr(self.c), _ptr(self.d), self.upsample, self.scale_main)


def quantize_multiplier(real: float) -> tuple[int, int]:
    m0 = ctypes.c_int32()
    sh = ctypes.c_int8()
    _check(load().aqd_quantize_multiplier(float(real), ctypes.byref(m0), ctypes.byref(sh)), "aqd_quantize_multiplier")
    return int(m0.value), int(sh.value)


class ConvWeights:
    """Prepared weights of one conv layer ([cout, kh, kw, cin] signed integers)."""

    def __init__(self, w_codes: torch.Tensor, w_bits: int, w_format: int = W_TWOS, stream=None):
        cout, kh, kw, cin = w_codes.shape
        packed = pack_codes(w_codes.reshape(-1, cin), w_bits, stream=stream)
        self._prepare(packed, cout, kh, kw, cin, w_bits, w_format, stream)

    @classmethod
    def from_packed(cls, packed: torch.Tensor, cout: int, kh: int, kw: int, cin: int, w_bits: int,
                    w_format: int = W_TWOS, stream=None) -> "ConvWeights":
        """packed: uint8 CUDA rows [cout*kh*kw, row_bytes(cin, w_bits)]."""
        self = cls.__new__(cls)
        self._prepare(packed.contiguous(), cout, kh, kw, cin, w_bits, w_format, stream)
        return self

    def _prepare(self, packed, cout, kh, kw, cin, w_bits, w_format, stream):
        L = load()
        nbytes = int(L.aqd_conv_weights_bytes(cout, kh, kw, cin))
        if nbytes == 0:
            raise ValueError("unsupported weight shape")
        self.buf = torch.zeros(nbytes + 256, dtype=torch.uint8, device=packed.device)
        off = (-self.buf.data_ptr()) % 256
        self.prepared = self.buf[off:off + nbytes]
        self.desc = _Weights(_ptr(self.prepared), cout, kh, kw, cin, w_bits, w_format)
        _check(L.aqd_conv_prepare_weights(_ptr(packed), ctypes.byref(self.desc), _ptr(self.prepared), nbytes,
                                          _stream(stream)), "aqd_conv_prepare_weights")
        self._packed = packed  # kept alive until the stream has consumed it
        self.cout, self.kh, self.kw, self.cin = cout, kh, kw, cin


def conv_out_hw(h, w, kh, kw, stride, pad):
    return (h + 2 * pad - kh) // stride + 1, (w + 2 * pad - kw) // stride + 1


def _ws(workspace: torch.Tensor | None):
    if workspace is None:
        return None, 0
    return _ptr(workspace), workspace.numel() * workspace.element_size()


def conv_int(x: DTensor, w: ConvWeights, stride: int, pad: int, y: DTensor, *, level: int = 0,
             rq: RequantParams | None = None, skip: DTensor | None = None, sp: SkipParams | None = None,
             workspace: torch.Tensor | None = None, stream=None) -> DTensor:
    xc, yc = x.ct(), y.ct()
    rqc = rq.c() if rq is not None else None
    skc = skip.ct() if skip is not None else None
    spc = sp.cs() if sp is not None else None
    wsp, wsb = _ws(workspace)
    _check(load().aqd_conv_int(ctypes.byref(xc), ctypes.byref(w.desc), stride, pad, level,
                               ctypes.byref(rqc) if rqc is not None else None,
                               ctypes.byref(skc) if skc is not None else None,
                               ctypes.byref(spc) if spc is not None else None, ctypes.byref(yc), wsp, wsb,
                               _stream(stream)),
           "aqd_conv_int")
    return y


def conv_int_static_workspace(x: DTensor, w: ConvWeights, stride: int, pad: int, y: DTensor, *, level: int = 0,
                              rq: RequantParams | None = None, skip: DTensor | None = None,
                              sp: SkipParams | None = None, stream=None) -> DTensor:
    """conv_int on the workspace path with the library's own fixed workspace (no allocation);
    calls that overlap in time share that workspace and must be ordered by the caller."""
    xc, yc = x.ct(), y.ct()
    rqc = rq.c() if rq is not None else None
    skc = skip.ct() if skip is not None else None
    spc = sp.cs() if sp is not None else None
    _check(load().aqd_conv_int_static_workspace(ctypes.byref(xc), ctypes.byref(w.desc), stride, pad, level,
                                                ctypes.byref(rqc) if rqc is not None else None,
                                                ctypes.byref(skc) if skc is not None else None,
                                                ctypes.byref(spc) if spc is not None else None, ctypes.byref(yc),
                                                _stream(stream)),
           "aqd_conv_int_static_workspace")
    return y


def _jobs(jobs):
    arr = (_Job * len(jobs))()
    for i, (x, y, skip, level) in enumerate(jobs):
        arr[i].x = x.ct()
        arr[i].y = y.ct() if y is not None else _Tensor(0, 0, 0, 0, 0, None)
        arr[i].skip = skip.ct() if skip is not None else _Tensor(0, 0, 0, 0, 0, None)
        arr[i].level = level
    return arr


def conv_workspace_bytes(jobs, w: ConvWeights, stride: int, pad: int) -> int:
    """Bytes of the expanded-activation workspace for these jobs (0: path not applicable)."""
    return int(load().aqd_conv_workspace_bytes(_jobs(jobs), len(jobs), ctypes.byref(w.desc), stride, pad))


def workspace_for(jobs, w: ConvWeights, stride: int, pad: int, device="cuda") -> torch.Tensor | None:
    """A 256-byte aligned workspace of the right size, or None when the path does not apply."""
    n = conv_workspace_bytes(jobs, w, stride, pad)
    if n == 0:
        return None
    buf = torch.empty(n + 256, dtype=torch.uint8, device=device)
    off = (-buf.data_ptr()) % 256
    return buf[off:off + n]


def conv_int_grouped(jobs, w: ConvWeights, stride: int, pad: int, *, rq: RequantParams | None = None,
                     sp: SkipParams | None = None, workspace: torch.Tensor | None = None, stream=None):
    """jobs: list of (x: DTensor, y: DTensor, skip: DTensor | None, level: int)."""
    arr = _jobs(jobs)
    rqc = rq.c() if rq is not None else None
    spc = sp.cs() if sp is not None else None
    wsp, wsb = _ws(workspace)
    _check(load().aqd_conv_int_grouped(arr, len(jobs), ctypes.byref(w.desc), stride, pad,
                                       ctypes.byref(rqc) if rqc is not None else None,
                                       ctypes.byref(spc) if spc is not None else None, wsp, wsb,
                                       _stream(stream)),
           "aqd_conv_int_grouped")


def conv_expand_input(jobs, w: ConvWeights, stride: int, pad: int, workspace: torch.Tensor, stream=None):
    """Only the expansion step of the workspace path: writes the zero-padded byte image of the
    jobs' inputs into `workspace` (jobs as for conv_int_grouped; y and skip are ignored)."""
    arr = _jobs(jobs)
    wsp, wsb = _ws(workspace)
    _check(load().aqd_conv_expand_input(arr, len(jobs), ctypes.byref(w.desc), stride, pad, wsp, wsb,
                                        _stream(stream)), "aqd_conv_expand_input")


def conv_int_grouped_expanded(jobs, w: ConvWeights, stride: int, pad: int, *, rq: RequantParams | None = None,
                              sp: SkipParams | None = None, workspace: torch.Tensor, stream=None):
    """conv_int_grouped fed from a workspace that already holds the expansion of these jobs'
    inputs (written by conv_expand_input); launches only the tensor-core convolution."""
    arr = _jobs(jobs)
    rqc = rq.c() if rq is not None else None
    spc = sp.cs() if sp is not None else None
    wsp, wsb = _ws(workspace)
    _check(load().aqd_conv_int_grouped_expanded(arr, len(jobs), ctypes.byref(w.desc), stride, pad,
                                                ctypes.byref(rqc) if rqc is not None else None,
                                                ctypes.byref(spc) if spc is not None else None, wsp, wsb,
                                                _stream(stream)),
           "aqd_conv_int_grouped_expanded")


def conv_int_grouped_chain(jobs, w: ConvWeights, stride: int, pad: int, *, rq: RequantParams | None = None,
                           sp: SkipParams | None = None, workspace: torch.Tensor, next_pad: int,
                           next_workspace: torch.Tensor, stream=None):
    """conv_int_grouped_expanded that also writes the outputs, one byte per code, as the
    zero-padded byte image the next stride-1 conv (padding next_pad) reads from
    next_workspace (whose border must hold zeros)."""
    arr = _jobs(jobs)
    rqc = rq.c() if rq is not None else None
    spc = sp.cs() if sp is not None else None
    wsp, wsb = _ws(workspace)
    nwp, nwb = _ws(next_workspace)
    _check(load().aqd_conv_int_grouped_chain(arr, len(jobs), ctypes.byref(w.desc), stride, pad,
                                             ctypes.byref(rqc) if rqc is not None else None,
                                             ctypes.byref(spc) if spc is not None else None, wsp, wsb,
                                             next_pad, nwp, nwb, _stream(stream)),
           "aqd_conv_int_grouped_chain")


def tower_sync_bytes(jobs, layers: int, pad: int) -> int:
    """Bytes of per-tile counters for conv_int_grouped_tower (jobs: layer 0's jobs)."""
    return int(load().aqd_conv_tower_sync_bytes(_jobs(jobs), len(jobs), layers, pad))


def conv_int_grouped_tower(layer_jobs, ws: list, rqs: list, pad: int, *, ws_a: torch.Tensor,
                           ws_b: torch.Tensor, sync: torch.Tensor | None, input_expanded: bool = False,
                           stream=None):
    """layer_jobs: one list of (x, y, None, level) per layer, layer i's x being layer i-1's y;
    ws: ConvWeights per layer; rqs: RequantParams per layer. See aqd_conv_int_grouped_tower."""
    nl, nj = len(layer_jobs), len(layer_jobs[0])
    arr = _jobs([jb for jobs in layer_jobs for jb in jobs])
    wd = (_Weights * nl)(*[w.desc for w in ws])
    rqa = (_Requant * nl)(*[r.c() for r in rqs])
    wap, wab = _ws(ws_a)
    wbp, wbb = _ws(ws_b)
    assert wab == wbb, "ws_a and ws_b must have the same size"
    sp_, sb = _ws(sync) if sync is not None else (None, 0)
    _check(load().aqd_conv_int_grouped_tower(arr, nj, nl, wd, rqa, pad, wap, wbp, wab, sp_, sb, int(input_expanded),
                                             _stream(stream)),
           "aqd_conv_int_grouped_tower")


def requant(acc: DTensor, rq: RequantParams, y: DTensor, *, level: int = 0, stream=None) -> DTensor:
    ac, yc, rqc = acc.ct(), y.ct(), rq.c()
    _check(load().aqd_requant(ctypes.byref(ac), ctypes.byref(rqc), level, ctypes.byref(yc), _stream(stream)),
           "aqd_requant")
    return y


def residual_add_int(a: DTensor, b: DTensor, sp: SkipParams, y: DTensor, *, rq: RequantParams | None = None,
                     level: int = 0, stream=None) -> DTensor:
    ac, bc, yc, spc = a.ct(), b.ct(), y.ct(), sp.cs()
    rqc = rq.c() if rq is not None else None
    _check(load().aqd_residual_add_int(ctypes.byref(ac), ctypes.byref(bc), ctypes.byref(spc),
                                       ctypes.byref(rqc) if rqc is not None else None, level, ctypes.byref(yc),
                                       _stream(stream)), "aqd_residual_add_int")
    return y


def maxpool_codes(x: DTensor, k: int, stride: int, pad: int, y: DTensor, stream=None) -> DTensor:
    xc, yc = x.ct(), y.ct()
    _check(load().aqd_maxpool_codes(ctypes.byref(xc), k, stride, pad, ctypes.byref(yc), _stream(stream)),
           "aqd_maxpool_codes")
    return y


def maxpool_expand(x: DTensor, k: int, stride: int, pad: int, y: DTensor, w: ConvWeights, conv_stride: int,
                   conv_pad: int, workspace: torch.Tensor, stream=None) -> DTensor:
    """maxpool_codes(x) -> y fused with conv_expand_input([(y, ...)], w, conv_stride, conv_pad,
    workspace): one pass writes y and the byte image of y for that convolution."""
    xc, yc = x.ct(), y.ct()
    wsp, wsb = _ws(workspace)
    _check(load().aqd_maxpool_expand(ctypes.byref(xc), k, stride, pad, ctypes.byref(yc), ctypes.byref(w.desc),
                                     conv_stride, conv_pad, wsp, wsb, _stream(stream)), "aqd_maxpool_expand")
    return y


def _f32(t: torch.Tensor | None):
    if t is None:
        return None
    if t.dtype != torch.float32 or not t.is_cuda or not t.is_contiguous():
        raise ValueError("expected a contiguous float32 CUDA tensor")
    return t.data_ptr()


def fake_quant(x: torch.Tensor, nu: float, bits: int, *, weight: bool = False, y: torch.Tensor | None = None,
               codes: torch.Tensor | None = None, stream=None):
    """Eq. 2 (weight=False) / Eq. 3 (weight=True) on a float32 tensor: returns (y, codes), the
    fake-quantized values and the uint8 codes (allocated when not given)."""
    y = torch.empty_like(x) if y is None else y
    codes = torch.empty(x.shape, dtype=torch.uint8, device=x.device) if codes is None else codes
    _check(load().aqd_fake_quant(_f32(x), x.numel(), float(nu), bits, int(weight), _f32(y), codes.data_ptr(),
                                 _stream(stream)), "aqd_fake_quant")
    return y, codes


def fake_quant_backward(x: torch.Tensor, gy: torch.Tensor, nu: float, bits: int, *, weight: bool = False,
                        gx: torch.Tensor | None = None, stream=None):
    """The STE backward of fake_quant: returns (gx, gnu) with gnu a one-element float64 CUDA
    tensor (the interval's gradient)."""
    gx = torch.empty_like(x) if gx is None else gx
    gnu = torch.empty(1, dtype=torch.float64, device=x.device)
    ws = torch.empty(int(load().aqd_fake_quant_backward_workspace_bytes()), dtype=torch.uint8, device=x.device)
    _check(load().aqd_fake_quant_backward(_f32(x), _f32(gy), x.numel(), float(nu), bits, int(weight), _f32(gx),
                                          gnu.data_ptr(), ws.data_ptr(), ws.numel(), _stream(stream)),
           "aqd_fake_quant_backward")
    return gx, gnu


def bn_level_stats(zs, stream=None):
    """Per-level batch mean and biased variance (float64 [levels, c]) of float32 CUDA tensors
    with channels last (Sec. 3.2.2's multi-level BN)."""
    c = zs[0].shape[-1]
    dev = zs[0].device
    nlev = len(zs)
    ptrs = (ctypes.c_void_p * nlev)(*[_f32(z) for z in zs])
    pix = (ctypes.c_int64 * nlev)(*[z.numel() // c for z in zs])
    mean = torch.empty((nlev, c), dtype=torch.float64, device=dev)
    var = torch.empty((nlev, c), dtype=torch.float64, device=dev)
    wsb = int(load().aqd_bn_level_stats_workspace_bytes(nlev, c))
    ws = torch.empty(max(wsb, 8), dtype=torch.uint8, device=dev)
    _check(load().aqd_bn_level_stats(ptrs, pix, nlev, c, mean.data_ptr(), var.data_ptr(), ws.data_ptr(), ws.numel(),
                                     _stream(stream)), "aqd_bn_level_stats")
    return mean, var


def device_status(stream=None) -> int:
    code = ctypes.c_int32()
    _check(load().aqd_device_status(_stream(stream), ctypes.byref(code)), "aqd_device_status")
    return int(code.value)


def selftest_wait_timeout(out: torch.Tensor, stream=None) -> None:
    """Launches the bounded-wait self-test into ``out`` (5 int64 on the device); see
    aqd_selftest_wait_timeout."""
    assert out.dtype == torch.int64 and out.is_cuda and out.numel() >= 5
    _check(load().aqd_selftest_wait_timeout(_ptr(out), _stream(stream)), "aqd_selftest_wait_timeout")


def set_conv_path(path: int) -> int:
    return int(load().aqd_set_conv_path(path))


def last_conv_path() -> int:
    return int(load().aqd_last_conv_path())
