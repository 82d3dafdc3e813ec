"""aqd_conv_int_grouped_tower: chained grouped layers whose launches overlap tile by tile
(each tile of layer i+1 waits, through per-tile counters, only for the tiles of layer i whose
rows it reads). Every output of every layer is compared with the oracle chain, for the full
RetinaNet head at 800x1333 (4 tower layers + the fused 256->84 cls/box conv), for level
widths whose dependency windows span more tiles (wp > 256), with the counters off and with
CTA pairs off (both run layer after layer), from a CUDA graph replayed several times, and
over calls back to back on one stream."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_same, to_device, weights
from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu


def _ref_conv(xt, wp, cv, level=0):
    return oracle.conv_int(xt, wp, cv.w_bits, 0, cv.kh, cv.kw, cv.stride, cv.pad, cv.cout, level=level,
                           m0=cv.m0, shift=cv.shift, bias=cv.bias,
                           levels=(cv.m0 if cv.m0 is not None else cv.bias).shape[0], out_bits=cv.out_bits)


class Tower:
    """The head as one tower call: tower layers, then cls and box fused as one 256->84 conv."""

    def __init__(self, wl, bits, ntower=4):
        self.wl, self.bits, self.nl = wl, bits, len(wl.inputs)
        self.xts = [oracle.CodeTensor.from_codes(x, bits) for x in wl.inputs]
        self.xs = [to_device(t) for t in self.xts]
        convs = wl.convs[:ntower]
        cls, box = wl.convs[4], wl.convs[5]
        self.tower = convs
        self.W = [weights(cv.w, bits) for cv in convs]
        self.Wh = weights(np.concatenate([cls.w, box.w]), bits)
        self.rqs = [aqd.RequantParams.from_numpy(cv.m0, cv.shift, cv.bias) for cv in convs]
        self.rqh = aqd.RequantParams.from_numpy(None, None, np.concatenate([cls.bias, box.bias], axis=1))
        self.ys = [[aqd.DTensor.empty(t.n, t.h, t.w, 256, bits) for t in self.xts] for _ in convs]
        self.heads = [aqd.DTensor.empty(t.n, t.h, t.w, cls.cout + box.cout, 32) for t in self.xts]
        ins = [self.xs] + self.ys
        self.layer_jobs = [[(ins[i][l], self.ys[i][l], None, l) for l in range(self.nl)] for i in range(len(convs))]
        self.layer_jobs.append([(ins[-1][l], self.heads[l], None, l) for l in range(self.nl)])
        self.ws_a = aqd.workspace_for(self.layer_jobs[0], self.W[0][0], 1, 1)
        self.ws_b = torch.zeros_like(self.ws_a)
        nbytes = aqd.tower_sync_bytes(self.layer_jobs[0], len(self.layer_jobs), 1)
        self.sync = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")

    def run(self, sync=True, stream=None):
        aqd.conv_int_grouped_tower(self.layer_jobs, [w for w, _ in self.W] + [self.Wh[0]], self.rqs + [self.rqh], 1,
                                   ws_a=self.ws_a, ws_b=self.ws_b, sync=self.sync if sync else None, stream=stream)

    def reference(self):
        refs = self.xts
        out = []
        for i, cv in enumerate(self.tower):
            refs = [_ref_conv(refs[l], self.W[i][1], cv, level=l) for l in range(self.nl)]
            out.append(refs)
        cls, box = self.wl.convs[4], self.wl.convs[5]
        heads = []
        for l in range(self.nl):
            hc = _ref_conv(refs[l], oracle.pack(cls.w.reshape(-1, cls.cin), self.bits), cls, level=l).codes()
            hb = _ref_conv(refs[l], oracle.pack(box.w.reshape(-1, box.cin), self.bits), box, level=l).codes()
            heads.append(np.concatenate([hc, hb], axis=-1))
        return out, heads

    def check(self, ref, what=""):
        out, heads = ref
        for i in range(len(self.tower)):
            for l in range(self.nl):
                assert_same(self.ys[i][l].data.cpu().numpy().reshape(out[i][l].packed.shape), out[i][l].packed, 256,
                            self.bits, f"{what} layer {i} level {l}")
        for l in range(self.nl):
            got = self.heads[l].data.cpu().numpy().view(np.int32).reshape(heads[l].shape)
            assert np.array_equal(got, heads[l]), f"{what} heads level {l}"


@pytest.mark.parametrize("calibrated", [False, True])
def test_full_head_tower_bit_exact(calibrated):
    t = Tower(synth.config2(calibrated=calibrated), 2)
    t.run()
    torch.cuda.synchronize()
    assert aqd.last_conv_path() == 6  # the 256->84 output conv on the FP4 pipe, from a nibble image
    assert aqd.device_status() == 0
    t.check(t.reference(), "full head")


@pytest.mark.parametrize("bits", [2, 3, 4])
def test_wide_levels_and_fallbacks_bit_exact(bits):
    """Level widths 300 and 600 (dependency windows of 5 and 7 tiles), a level narrower than a
    tile, batch 2; then the same with the counters off, with CTA pairs off, and with the FP4
    pipe off (the output conv then reads a byte image on the E4M3 pipe)."""
    levels = [(7, 300), (5, 600), (9, 20), (1, 3)]
    wl = synth.head_tower(60 + bits, 2, bits, levels=levels, calibrated=True)
    t = Tower(wl, bits, ntower=3)
    ref = t.reference()
    t.run()
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    t.check(ref, "overlapped")
    for mode in ("no sync", "no pairs", "no fp4"):
        for ys in t.ys:
            for y in ys:
                y.data.fill_(0xEE)
        old = aqd.set_conv_path({"no pairs": 3, "no fp4": 4}.get(mode, 0))
        try:
            t.run(sync=mode != "no sync")
        finally:
            aqd.set_conv_path(old)
        torch.cuda.synchronize()
        assert aqd.device_status() == 0
        t.check(ref, mode)


def test_graph_replays_and_back_to_back_calls():
    """The tower captured in a CUDA graph (the counter reset is a node of it) and replayed
    five times, with the inputs changed between replays; then ten calls back to back on one
    stream, the last one's outputs compared."""
    levels = [(20, 34), (10, 17), (5, 9), (3, 5), (2, 3)]
    wl = synth.head_tower(71, 2, 2, levels=levels, calibrated=True)
    t = Tower(wl, 2)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        t.run(stream=s)
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        t.run(stream=s)
    rng = np.random.default_rng(5)
    for rep in range(5):
        new = [synth.act_codes(rng, x.shape, 2) for x in wl.inputs]
        t.xts = [oracle.CodeTensor.from_codes(x, 2) for x in new]
        for d, h in zip(t.xs, t.xts):
            d.data.copy_(torch.from_numpy(h.packed).reshape(d.data.shape))
        with torch.cuda.stream(s):
            g.replay()
        s.synchronize()
        if rep in (0, 4):
            t.check(t.reference(), f"replay {rep}")
    with torch.cuda.stream(s):
        for _ in range(10):
            t.run(stream=s)
    s.synchronize()
    assert aqd.device_status() == 0
    t.check(t.reference(), "back to back")


def test_tower_argument_errors():
    levels = [(20, 34)]  # three tiles per layer: the two fused tower layers need 12 bytes of counters
    wl = synth.head_tower(72, 1, 2, levels=levels, calibrated=True)
    t = Tower(wl, 2, ntower=2)
    # layer 1's input is not layer 0's output
    bad = [list(j) for j in t.layer_jobs]
    bad[1][0] = (t.xs[0], t.ys[1][0], None, 0)
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int_grouped_tower(bad, [w for w, _ in t.W] + [t.Wh[0]], t.rqs + [t.rqh], 1, ws_a=t.ws_a,
                                   ws_b=t.ws_b, sync=t.sync)
    assert e.value.status == 1
    # counters too small (4 of the 12 bytes)
    assert aqd.tower_sync_bytes(t.layer_jobs[0], 2, 1) == 12
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int_grouped_tower(t.layer_jobs, [w for w, _ in t.W] + [t.Wh[0]], t.rqs + [t.rqh], 1,
                                   ws_a=t.ws_a, ws_b=t.ws_b, sync=t.sync[:4])
    assert e.value.status == 1
