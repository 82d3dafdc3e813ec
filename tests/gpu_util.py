"""Helpers of the GPU parity tests: run one step on libaqd (through the C ABI) and the
same step on the CPU oracle from identical seeded inputs, and compare bytes.

Inputs are packed by the oracle's own packer and copied to the device, so the CUDA path
never produces an oracle input."""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2007_06919_gb300 import aqd


def dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def to_device(t: oracle.CodeTensor) -> aqd.DTensor:
    return aqd.DTensor(dev(t.packed), t.n, t.h, t.w, t.c, t.bits)


def weights(w_codes: np.ndarray, w_bits: int, w_format: int = 0):
    """Prepared GPU weights from oracle-packed bytes, plus the packed bytes for the oracle."""
    cout, kh, kw, cin = w_codes.shape
    packed = oracle.pack(w_codes.reshape(-1, cin), w_bits)
    return aqd.ConvWeights.from_packed(dev(packed), cout, kh, kw, cin, w_bits, w_format), packed


def conv_pair(x: np.ndarray, x_bits: int, w: np.ndarray, w_bits: int, *, w_format: int = 0, stride: int = 1,
              pad: int = 1, out_bits: int = 2, m0=None, shift=None, bias=None, level: int = 0,
              skip: np.ndarray | None = None, skip_bits: int = 4, skip_c=None, skip_d=None, upsample: int = 1,
              scale_main: int = 0, path: int = 0, wprep=None, workspace: bool = False):
    """Returns (gpu_bytes, oracle_bytes, used_path) for one convolution. With workspace=True
    the call gets an expanded-activation workspace when that path applies."""
    n, h, wd, cin = x.shape
    cout, kh, kw, _ = w.shape
    xt = oracle.CodeTensor.from_codes(x, x_bits)
    W, wp = wprep if wprep is not None else weights(w, w_bits, w_format)
    levels = (m0 if m0 is not None else bias).shape[0] if (m0 is not None or bias is not None) else 1
    skt = oracle.CodeTensor.from_codes(skip, skip_bits) if skip is not None else None
    ref = oracle.conv_int(xt, wp, w_bits, w_format, kh, kw, stride, pad, cout, level=level, m0=m0, shift=shift,
                          bias=bias, levels=levels, skip=skt, skip_c=skip_c, skip_d=skip_d, upsample=upsample,
                          scale_main=scale_main, out_bits=out_bits)
    X = to_device(xt)
    Y = aqd.DTensor.empty(ref.n, ref.h, ref.w, cout, out_bits)
    Y.data.fill_(0xA5)  # poison: every output byte must be written
    rq = aqd.RequantParams.from_numpy(m0, shift, bias) if (m0 is not None or bias is not None) else None
    S = to_device(skt) if skt is not None else None
    sp = aqd.SkipParams.from_numpy(skip_c, skip_d, upsample, scale_main) if skip is not None else None
    ws = aqd.workspace_for([(X, Y, S, level)], W, stride, pad) if workspace else None
    if ws is not None:
        ws.fill_(0x5A)  # stale contents must not matter
    old = aqd.set_conv_path(path)
    try:
        aqd.conv_int(X, W, stride, pad, Y, level=level, rq=rq, skip=S, sp=sp, workspace=ws)
        used = aqd.last_conv_path()
    finally:
        aqd.set_conv_path(old)
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    return Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, used


def assert_same(got: np.ndarray, want: np.ndarray, c: int, bits: int, what: str = ""):
    if np.array_equal(got, want):
        return
    g = oracle.unpack(got, c, bits) if bits != 32 else got.view(np.int32)
    r = oracle.unpack(want, c, bits) if bits != 32 else want.view(np.int32)
    bad = np.argwhere(g != r)
    raise AssertionError(f"{what}: {len(bad)} of {g.size} values differ; first at {bad[:5].tolist()}: "
                         f"gpu {g[tuple(bad[0])]} oracle {r[tuple(bad[0])]}")
