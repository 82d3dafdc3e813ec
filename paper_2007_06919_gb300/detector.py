"""The whole integer-only detector (integer ResNet-18 + FPN + shared RetinaNet head) on the
GPU: a network given as a list of layers (convs and code max-pools naming their input,
output and skip tensors) runs as a fixed sequence of libaqd launches on one stream.

Every conv is one grouped call (the head's five FPN levels in one launch, each with its own
row of the per-level tables, Sec. 3.2.2); skips (identity codes, int32 downsample branches,
the FPN's nearest-2x top-down maps) are added in the conv epilogue (Eq. 7). Output tensors
and one shared expanded-activation workspace are allocated once, up front, so the whole
forward pass can be captured in a CUDA graph.

Three launch-level fusions, none of which changes any output value:
- the classification (256->80) and box (256->4) convs read the same tower output, so they run
  as one 256->84 conv with concatenated weight rows and biases (``fuse_heads``);
- a stride-1 conv whose only consumer is a stride-1 conv on the workspace path writes that
  consumer's zero-padded byte image in its epilogue (``chain``), so the consumer skips the
  expansion pass. The head tower uses it: the image of tower layer i is the input of i+1;
- a max-pool on codes whose output the next conv reads on the workspace path (the stem's
  3x3 stride-2 pool and the first residual stage) runs inside that conv's expansion pass
  (``fuse_pool``, aqd_maxpool_expand): the pooled codes are still written for the stage's
  skip, but not read back for the expansion, and the pool launch disappears.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

from . import aqd


@dataclass
class _ConvPlan:
    layer: object
    w: aqd.ConvWeights
    rq: aqd.RequantParams | None
    sp: aqd.SkipParams | None
    jobs: list
    stride: int
    pad: int
    ws_bytes: int          # expanded-activation bytes of this conv (0: in-kernel path)
    reads_image: bool = False   # input image already written by the producer (chained)
    chain_to: "_ConvPlan | None" = None
    image: int = 0         # which of the two chain images this conv reads (when reads_image)
    pool: object = None    # the max-pool layer fused into this conv's expansion pass


def _aligned(nbytes: int, device) -> torch.Tensor:
    buf = torch.zeros(nbytes + 256, dtype=torch.uint8, device=device)
    off = (-buf.data_ptr()) % 256
    return buf[off:off + nbytes]


class IntDetector:
    """Plans and runs a layer list on one GPU.

    layers: the network (each with ``name``, ``src``, ``dst``, ``conv`` or ``pool``, ``skip``,
    ``upsample``), in execution order. image_shape: (n, h, w, c, bits) of the input tensor,
    named "image". The caller writes the input codes into ``self.tensors["image"]`` (or passes
    a DTensor of that shape to ``forward``)."""

    def __init__(self, layers, image_shape, device="cuda", fuse_heads: bool = True, chain: bool = True,
                 fuse_pool: bool = True):
        self.device = torch.device(device)
        n, h, w, c, bits = image_shape
        self.tensors: dict[str, aqd.DTensor] = {"image": aqd.DTensor.empty(n, h, w, c, bits, device=self.device)}
        self.steps = []           # ("pool", layer) or ("conv", _ConvPlan)
        self.fused = {}           # fused output name -> (first name, second name, first's channels)
        self.ops = 0              # 2*M*N*K over all convs (the real, unpadded work)
        layers = list(layers)
        if fuse_heads:
            layers = self._fuse_output_convs(layers)
        ws_max = 0
        for ly in layers:
            if ly.pool is not None:
                k, s, p = ly.pool
                x = self.tensors[ly.src[0]]
                ho, wo = aqd.conv_out_hw(x.h, x.w, k, k, s, p)
                self.tensors[ly.dst[0]] = aqd.DTensor.empty(x.n, ho, wo, x.c, x.bits, device=self.device)
                self.steps.append(("pool", ly))
                continue
            cv = ly.conv
            for src, dst in zip(ly.src, ly.dst):
                x = self.tensors[src]
                ho, wo = aqd.conv_out_hw(x.h, x.w, cv.kh, cv.kw, cv.stride, cv.pad)
                self.tensors[dst] = aqd.DTensor.empty(x.n, ho, wo, cv.cout, cv.out_bits, device=self.device)
                self.ops += 2 * x.n * ho * wo * cv.cout * cv.kh * cv.kw * cv.cin
            W = aqd.ConvWeights(torch.from_numpy(np.ascontiguousarray(cv.w)).to(self.device), cv.w_bits)
            rq = None
            if cv.m0 is not None or cv.bias is not None:
                rq = aqd.RequantParams.from_numpy(cv.m0, cv.shift, cv.bias, device=self.device)
            sp = None
            if ly.skip:
                sp = aqd.SkipParams.from_numpy(cv.skip_c, cv.skip_d, ly.upsample, 0, device=self.device)
            jobs = [(self.tensors[s], self.tensors[d], self.tensors[k] if ly.skip else None, l)
                    for l, (s, d, k) in enumerate(zip(ly.src, ly.dst, ly.skip or [None] * len(ly.src)))]
            wsb = aqd.conv_workspace_bytes(jobs, W, cv.stride, cv.pad)
            ws_max = max(ws_max, wsb)
            self.steps.append(("conv", _ConvPlan(ly, W, rq, sp, jobs, cv.stride, cv.pad, wsb)))
        if chain:
            self._plan_chains(layers)
        if fuse_pool:
            self._plan_pool_fusion()
        self.workspace = _aligned(ws_max, self.device) if ws_max else None
        # byte images of chained convs, two per geometry (conv i writes the one conv i+1 reads);
        # their zero borders are written here once and never touched again
        self.images = {}
        for k, p in self.steps:
            if k == "conv" and p.reads_image and self._image_key(p) not in self.images:
                self.images[self._image_key(p)] = [_aligned(p.ws_bytes, self.device) for _ in range(2)]
        # a conv that expands its own input is two launches (with a fused pool the expansion
        # launch is the pool's, whose own step is gone)
        self.launches = sum(1 + (1 if (k == "conv" and p.ws_bytes and not p.reads_image) else 0)
                            for k, p in self.steps)

    # -------------------------------------------------------------- planning

    def _fuse_output_convs(self, layers):
        """Two int32 convs with the same inputs, geometry and bias-only epilogue (the cls and
        box heads) become one conv over the concatenated output channels; ``self.fused`` maps
        each fused output name to (first name, second name, channels of the first)."""
        from copy import copy
        out = []
        i = 0
        while i < len(layers):
            a = layers[i]
            b = layers[i + 1] if i + 1 < len(layers) else None
            if (b is not None and a.conv is not None and b.conv is not None and a.src == b.src
                    and not a.skip and not b.skip and a.conv.out_bits == 32 and b.conv.out_bits == 32
                    and a.conv.m0 is None and b.conv.m0 is None
                    and (a.conv.kh, a.conv.kw, a.conv.stride, a.conv.pad, a.conv.cin, a.conv.w_bits)
                    == (b.conv.kh, b.conv.kw, b.conv.stride, b.conv.pad, b.conv.cin, b.conv.w_bits)):
                cv = copy(a.conv)
                cv.w = np.concatenate([a.conv.w, b.conv.w])
                cv.bias = np.concatenate([a.conv.bias, b.conv.bias], axis=1)
                cv.cout = a.conv.cout + b.conv.cout
                ly = copy(a)
                ly.name = f"{a.name}+{b.name}"
                ly.conv = cv
                ly.dst = [f"{x}+{y}" for x, y in zip(a.dst, b.dst)]
                for f, x, y in zip(ly.dst, a.dst, b.dst):
                    self.fused[f] = (x, y, a.conv.cout)
                out.append(ly)
                i += 2
                continue
            out.append(a)
            i += 1
        return out

    def _plan_chains(self, layers):
        """Marks producer -> consumer pairs that hand over the byte image directly: the consumer
        is the next conv, reads exactly the producer's outputs (same job order), and both are
        stride-1 convs on the workspace path; the producer writes 2- to 4-bit codes in blocks of
        64 channels. The producer still writes its packed outputs for any other reader."""
        convs = [p for k, p in self.steps if k == "conv"]
        for a, b in zip(convs, convs[1:]):
            ca, cb = a.layer.conv, b.layer.conv
            if (list(b.layer.src) == list(a.layer.dst) and b.ws_bytes and a.ws_bytes
                    and ca.stride == 1 and cb.stride == 1 and 2 <= ca.out_bits <= 4 and ca.cout % 64 == 0):
                a.chain_to = b
                b.reads_image = True
        # chained images are keyed by geometry (input shapes and padding): the zero border of
        # an image is written once, so one buffer never serves two geometries; along a chain
        # the consumer reads the other buffer of the pair than its producer
        for p in convs:
            if p.chain_to is not None:
                p.chain_to.image = 1 - p.image if p.reads_image else 0

    def _plan_pool_fusion(self):
        """Marks 3x3 stride-2 max-pools on 2- or 4-bit codes whose output is the single input of
        the next step, a conv on the workspace path that expands its own input (not chained):
        that conv's expansion pass computes the pool (aqd_maxpool_expand)."""
        for (k0, ly), (k1, p) in zip(self.steps, self.steps[1:]):
            if (k0 == "pool" and k1 == "conv" and p.ws_bytes and not p.reads_image
                    and tuple(ly.pool[:2]) == (3, 2) and list(p.layer.src) == [ly.dst[0]]
                    and self.tensors[ly.dst[0]].bits in (2, 4)):
                p.pool = ly
        fused = {id(p.pool) for k, p in self.steps if k == "conv" and p.pool is not None}
        self.steps = [(k, p) for k, p in self.steps if not (k == "pool" and id(p) in fused)]

    @staticmethod
    def _image_key(p: _ConvPlan):
        return (tuple((x.n, x.h, x.w, x.c) for x, _, _, _ in p.jobs), p.pad, p.ws_bytes)

    # -------------------------------------------------------------- running

    def forward(self, image: aqd.DTensor | None = None, stream=None):
        """Enqueues the whole network on ``stream`` (the current stream if None)."""
        T = self.tensors
        if image is not None and image.data.data_ptr() != T["image"].data.data_ptr():
            T["image"].data.copy_(image.data)
        for kind, p in self.steps:
            if kind == "pool":
                k, s, pd = p.pool
                aqd.maxpool_codes(T[p.src[0]], k, s, pd, T[p.dst[0]], stream=stream)
                continue
            if p.reads_image:
                src_ws = self.images[self._image_key(p)][p.image]
            else:
                src_ws = self.workspace[:p.ws_bytes] if p.ws_bytes else None
            if p.pool is not None:
                k, s, pd = p.pool.pool
                aqd.maxpool_expand(T[p.pool.src[0]], k, s, pd, T[p.pool.dst[0]], p.w, p.stride, p.pad, src_ws,
                                   stream=stream)
            if p.chain_to is not None:
                nxt = p.chain_to
                if not p.reads_image and p.pool is None:
                    aqd.conv_expand_input(p.jobs, p.w, p.stride, p.pad, src_ws, stream=stream)
                aqd.conv_int_grouped_chain(p.jobs, p.w, p.stride, p.pad, rq=p.rq, sp=p.sp, workspace=src_ws,
                                           next_pad=nxt.pad, next_workspace=self.images[self._image_key(nxt)][nxt.image],
                                           stream=stream)
            elif p.reads_image or p.pool is not None:
                aqd.conv_int_grouped_expanded(p.jobs, p.w, p.stride, p.pad, rq=p.rq, sp=p.sp, workspace=src_ws,
                                              stream=stream)
            else:
                aqd.conv_int_grouped(p.jobs, p.w, p.stride, p.pad, rq=p.rq, sp=p.sp, workspace=src_ws,
                                     stream=stream)
        return T

    def output(self, name: str) -> torch.Tensor:
        """A layer output as int32 codes [n, h, w, c]; for convs that ran fused ("cls.l" and
        "box.l") the channel slice of the fused tensor."""
        if name in self.tensors:
            return self.tensors[name].codes()
        for f, (a, b, ca) in self.fused.items():
            if name == a:
                return self.tensors[f].codes()[..., :ca]
            if name == b:
                return self.tensors[f].codes()[..., ca:]
        raise KeyError(name)
