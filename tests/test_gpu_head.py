"""GPU parity at the workloads' full sizes: the ResNet-50 C3 bottleneck (4-bit, identity
skip), the shared RetinaNet head tower over the five FPN levels with multi-level BN tables
(2-bit, grouped launch), and the 2/3/4/8-bit sweep of that tower at batch 16."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_same, dev, to_device, weights
from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu


def _ref_conv(xt, wp, cv, level=0, skip=None):
    return oracle.conv_int(xt, wp, cv.w_bits, 0, cv.kh, cv.kw, cv.stride, cv.pad, cv.cout, level=level,
                           m0=cv.m0, shift=cv.shift, bias=cv.bias,
                           levels=(cv.m0 if cv.m0 is not None else cv.bias).shape[0], skip=skip,
                           skip_c=cv.skip_c, skip_d=cv.skip_d, out_bits=cv.out_bits)


def _rq(cv):
    return aqd.RequantParams.from_numpy(cv.m0, cv.shift, cv.bias)


@pytest.mark.parametrize("ws", [False, True])
def test_config1_bottleneck_chain_bit_exact(ws):
    """1x1 512->128, 3x3 128->128, 1x1 128->512 + identity skip (Eq. 7), all at
    2 x 100 x 152, 4-bit: each stage is compared; the GPU chain feeds itself and the
    oracle chain feeds itself."""
    wl = synth.config1()
    x = wl.inputs[0]
    xt = oracle.CodeTensor.from_codes(x, 4)
    ref = xt
    cur = to_device(xt)
    for i, cv in enumerate(wl.convs):
        W, wp = weights(cv.w, 4)
        skip_ref = xt if cv.skip_c is not None else None
        ref = _ref_conv(ref, wp, cv, skip=skip_ref)
        Y = aqd.DTensor.empty(ref.n, ref.h, ref.w, cv.cout, 4)
        sp = aqd.SkipParams.from_numpy(cv.skip_c, cv.skip_d) if cv.skip_c is not None else None
        skt = to_device(xt) if sp else None
        wsb = aqd.workspace_for([(cur, Y, skt, 0)], W, cv.stride, cv.pad) if ws else None
        aqd.conv_int(cur, W, cv.stride, cv.pad, Y, rq=_rq(cv), skip=skt, sp=sp, workspace=wsb)
        assert aqd.last_conv_path() == (4 if ws else 1)
        torch.cuda.synchronize()
        assert_same(Y.data.cpu().numpy().reshape(ref.packed.shape), ref.packed, cv.cout, 4, f"stage {i}")
        cur = Y
    assert aqd.device_status() == 0
    assert len(np.unique(ref.codes())) > 3


def _tower_levels_gpu(inputs, convs, bits, grouped=True, ws=False):
    """Runs the 4-layer tower + cls/box on every level; returns per-level outputs."""
    nl = len(inputs)
    xs = [to_device(oracle.CodeTensor.from_codes(x, bits)) for x in inputs]
    for cv in convs[:4]:
        W, _ = weights(cv.w, bits)
        ys = [aqd.DTensor.empty(x.n, x.h, x.w, 256, bits) for x in xs]
        if grouped:
            jobs = [(xs[l], ys[l], None, l) for l in range(nl)]
            wsb = aqd.workspace_for(jobs, W, 1, 1) if ws else None
            aqd.conv_int_grouped(jobs, W, 1, 1, rq=_rq(cv), workspace=wsb)
            assert aqd.last_conv_path() == (4 if ws else 1)
        else:
            for l in range(nl):
                aqd.conv_int(xs[l], W, 1, 1, ys[l], level=l, rq=_rq(cv))
        xs = ys
    heads = []
    for cv in convs[4:]:
        W, _ = weights(cv.w, bits)
        ys = [aqd.DTensor.empty(x.n, x.h, x.w, cv.cout, 32) for x in xs]
        jobs = [(xs[l], ys[l], None, l) for l in range(nl)]
        wsb = aqd.workspace_for(jobs, W, 1, 1) if ws else None
        aqd.conv_int_grouped(jobs, W, 1, 1, rq=aqd.RequantParams.from_numpy(None, None, cv.bias), workspace=wsb)
        heads.append(ys)
    torch.cuda.synchronize()
    return xs, heads


def _tower_levels_ref(inputs, convs, bits):
    xs = [oracle.CodeTensor.from_codes(x, bits) for x in inputs]
    for cv in convs[:4]:
        wp = oracle.pack(cv.w.reshape(-1, cv.cin), bits)
        xs = [_ref_conv(xs[l], wp, cv, level=l) for l in range(len(xs))]
    heads = []
    for cv in convs[4:]:
        wp = oracle.pack(cv.w.reshape(-1, cv.cin), bits)
        heads.append([_ref_conv(xs[l], wp, cv, level=l) for l in range(len(xs))])
    return xs, heads


@pytest.mark.parametrize("calibrated,ws", [(False, False), (True, False), (False, True), (True, True)])
def test_head_tower_full_size_bit_exact(calibrated, ws):
    """The whole detector head at 800x1333 (levels 100x168 .. 7x11), batch 2, 2-bit:
    4 grouped tower layers + cls (80) + box (4) int32 heads, every output compared."""
    wl = synth.config2(calibrated=calibrated)
    g_tower, g_heads = _tower_levels_gpu(wl.inputs, wl.convs, 2, ws=ws)
    r_tower, r_heads = _tower_levels_ref(wl.inputs, wl.convs, 2)
    for l in range(5):
        assert_same(g_tower[l].data.cpu().numpy().reshape(r_tower[l].packed.shape), r_tower[l].packed, 256, 2,
                    f"tower level {l}")
        for hi, cout in enumerate((80, 4)):
            assert_same(g_heads[hi][l].data.cpu().numpy().reshape(r_heads[hi][l].packed.shape),
                        r_heads[hi][l].packed, cout, 32, f"head {cout} level {l}")
    assert aqd.device_status() == 0
    if calibrated:
        assert len(np.unique(r_tower[0].codes())) == 4


def test_grouped_launch_equals_per_level_launches():
    wl = synth.head_tower(9, 2, 2, levels=[(20, 34), (10, 17), (5, 9), (3, 5), (2, 3)], calibrated=True)
    a, ah = _tower_levels_gpu(wl.inputs, wl.convs, 2, grouped=True, ws=True)
    b, bh = _tower_levels_gpu(wl.inputs, wl.convs, 2, grouped=False)
    for l in range(5):
        assert torch.equal(a[l].data, b[l].data)
        assert torch.equal(ah[0][l].data, bh[0][l].data)


@pytest.mark.parametrize("bits", [2, 3, 4, 8])
def test_bitwidth_sweep_batch16_bit_exact(bits):
    """First tower layer of the batch-16 head for each bit width (config 4), all five levels in
    one grouped launch (on the expanded-activation workspace; 8-bit codes split into 4-bit
    halves on the tensor cores): every output byte of every level against the oracle's full
    convolution (about 423 GOP per bit width on the host cores)."""
    wl = synth.config4(bits)
    cv = wl.convs[0]
    W, wp = weights(cv.w, bits)
    xts = [oracle.CodeTensor.from_codes(x, bits) for x in wl.inputs]
    xs = [to_device(t) for t in xts]
    ys = [aqd.DTensor.empty(x.n, x.h, x.w, 256, bits) for x in xs]
    for y in ys:
        y.data.fill_(0xA5)
    jobs = [(xs[l], ys[l], None, l) for l in range(5)]
    wsb = aqd.workspace_for(jobs, W, 1, 1)
    aqd.conv_int_grouped(jobs, W, 1, 1, rq=_rq(cv), workspace=wsb)
    assert aqd.last_conv_path() == 4
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    for l in range(5):
        want = oracle.conv_int(xts[l], wp, bits, 0, 3, 3, 1, 1, 256, level=l, m0=cv.m0, shift=cv.shift,
                               bias=cv.bias, levels=5, out_bits=bits)
        got = ys[l].data.cpu().numpy().reshape(want.packed.shape)
        assert_same(got, want.packed, 256, bits, f"config 4, {bits}-bit, level {l}")


def test_cls_and_box_as_one_conv_bit_exact():
    """The benchmark's fused output conv: the 256->80 classification and 256->4 box weights
    (and biases) concatenated into one 256->84 conv over the same tower output; channels
    0..79 and 80..83 must equal the two separate convs of the oracle on every level."""
    wl = synth.head_tower(11, 2, 2, levels=[(20, 34), (10, 17), (5, 9), (3, 5), (2, 3)], calibrated=True)
    cls, box = wl.convs[4:]
    rng = np.random.default_rng(11)
    xts = [oracle.CodeTensor.from_codes(synth.act_codes(rng, x.shape[:3] + (256,), 2), 2) for x in wl.inputs]
    W, _ = weights(np.concatenate([cls.w, box.w]), 2)
    rq = aqd.RequantParams.from_numpy(None, None, np.concatenate([cls.bias, box.bias], axis=1))
    xs = [to_device(t) for t in xts]
    ys = [aqd.DTensor.empty(t.n, t.h, t.w, 84, 32) for t in xts]
    jobs = [(xs[l], ys[l], None, l) for l in range(5)]
    aqd.conv_int_grouped(jobs, W, 1, 1, rq=rq, workspace=aqd.workspace_for(jobs, W, 1, 1))
    assert aqd.last_conv_path() == 6  # 2-bit codes, 84 channels: the FP4 pipe
    torch.cuda.synchronize()
    for l in range(5):
        got = ys[l].data.cpu().numpy().view(np.int32).reshape(-1, 84)
        for cv, lo in ((cls, 0), (box, 80)):
            wp = oracle.pack(cv.w.reshape(-1, cv.cin), 2)
            want = _ref_conv(xts[l], wp, cv, level=l).packed.view(np.int32).reshape(-1, cv.cout)
            assert np.array_equal(got[:, lo:lo + cv.cout], want), f"level {l} head {cv.cout}"
    assert aqd.device_status() == 0


def test_expand_once_then_two_convs_bit_exact():
    """aqd_conv_expand_input once, then aqd_conv_int_grouped_expanded twice from the same
    workspace (the classification and box convs over one tower output, levels grouped):
    both must equal the oracle; the tower conv from the split calls must equal the
    one-call grouped conv byte for byte."""
    levels = [(16, 27), (8, 14), (4, 7)]
    wl = synth.head_tower(31, 2, 2, levels=levels, calibrated=True)
    tower, cls, box = wl.convs[0], wl.convs[4], wl.convs[5]
    xts = [oracle.CodeTensor.from_codes(x, 2) for x in wl.inputs]
    xs = [to_device(t) for t in xts]
    Wt, _ = weights(tower.w, 2)
    y1 = [aqd.DTensor.empty(t.n, t.h, t.w, 256, 2) for t in xts]
    y2 = [aqd.DTensor.empty(t.n, t.h, t.w, 256, 2) for t in xts]
    jobs1 = [(xs[l], y1[l], None, l) for l in range(3)]
    jobs2 = [(xs[l], y2[l], None, l) for l in range(3)]
    ws = aqd.workspace_for(jobs1, Wt, 1, 1)
    aqd.conv_int_grouped(jobs1, Wt, 1, 1, rq=_rq(tower), workspace=ws)
    ws.fill_(0x5A)
    aqd.conv_expand_input(jobs2, Wt, 1, 1, ws)
    aqd.conv_int_grouped_expanded(jobs2, Wt, 1, 1, rq=_rq(tower), workspace=ws)
    assert aqd.last_conv_path() == 4
    torch.cuda.synchronize()
    for l in range(3):
        assert torch.equal(y1[l].data, y2[l].data), f"tower level {l}"
    # two convs from one expansion of the tower output
    ws2 = aqd.workspace_for([(y1[l], y1[l], None, l) for l in range(3)], Wt, 1, 1)
    aqd.conv_expand_input([(y1[l], None, None, l) for l in range(3)], Wt, 1, 1, ws2)
    outs = {}
    for cv in (cls, box):
        W, _ = weights(cv.w, 2)
        ys = [aqd.DTensor.empty(t.n, t.h, t.w, cv.cout, 32) for t in xts]
        aqd.conv_int_grouped_expanded([(y1[l], ys[l], None, l) for l in range(3)], W, 1, 1,
                                      rq=aqd.RequantParams.from_numpy(None, None, cv.bias), workspace=ws2)
        outs[cv.cout] = ys
    torch.cuda.synchronize()
    wpt = oracle.pack(tower.w.reshape(-1, tower.cin), 2)
    for l in range(3):
        mid = _ref_conv(xts[l], wpt, tower, level=l)  # the oracle's own tower output
        assert_same(y1[l].data.cpu().numpy().reshape(mid.packed.shape), mid.packed, 256, 2, f"tower {l}")
        for cv in (cls, box):
            wp = oracle.pack(cv.w.reshape(-1, cv.cin), 2)
            want = _ref_conv(mid, wp, cv, level=l).packed
            assert_same(outs[cv.cout][l].data.cpu().numpy().reshape(want.shape), want, cv.cout, 32,
                        f"head {cv.cout} level {l}")
    assert aqd.device_status() == 0


def test_expanded_conv_needs_an_applicable_workspace():
    rng = np.random.default_rng(3)
    W, _ = weights(synth.weight_codes(rng, (64, 3, 3, 96), 2), 2)  # cin 96: no workspace path
    X = aqd.DTensor.empty(1, 8, 8, 96, 2)
    Y = aqd.DTensor.empty(1, 8, 8, 64, 32)
    buf = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int_grouped_expanded([(X, Y, None, 0)], W, 1, 1, workspace=buf)
    assert e.value.status == 1
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_expand_input([(X, Y, None, 0)], W, 1, 1, buf)
    assert e.value.status == 1


@pytest.mark.parametrize("bits,pairs", [(2, True), (2, False), (3, True), (4, True)])
def test_chained_tower_bit_exact(bits, pairs):
    """Layer chaining: the input expanded once, then three tower layers each written by
    aqd_conv_int_grouped_chain straight into the next layer's byte image (two workspaces
    in turn, the second zero-filled once), then the output conv from the last image. Every
    layer's packed output equals the oracle chain's, and every chained image equals what
    aqd_conv_expand_input writes for that layer's output."""
    levels = [(15, 26), (8, 13), (4, 7)]
    wl = synth.head_tower(41 + bits, 2, bits, levels=levels, calibrated=True)
    nl = len(levels)
    xts = [oracle.CodeTensor.from_codes(x, bits) for x in wl.inputs]
    xs = [to_device(t) for t in xts]
    Ws = [weights(cv.w, bits) for cv in wl.convs]
    old = aqd.set_conv_path(1 if pairs else 3)
    try:
        jobs0 = [(xs[l], None, None, l) for l in range(nl)]
        wsA = aqd.workspace_for(jobs0, Ws[0][0], 1, 1)
        wsB = torch.zeros_like(wsA)
        wsA.fill_(0x5A)
        aqd.conv_expand_input(jobs0, Ws[0][0], 1, 1, wsA)
        cur_ws, nxt_ws = wsA, wsB
        cur = xs
        refs = xts
        for i in range(3):
            cv = wl.convs[i]
            ys = [aqd.DTensor.empty(t.n, t.h, t.w, 256, bits) for t in refs]
            jobs = [(cur[l], ys[l], None, l) for l in range(nl)]
            aqd.conv_int_grouped_chain(jobs, Ws[i][0], 1, 1, rq=_rq(cv), workspace=cur_ws, next_pad=1,
                                       next_workspace=nxt_ws)
            torch.cuda.synchronize()
            refs = [_ref_conv(refs[l], Ws[i][1], cv, level=l) for l in range(nl)]
            for l in range(nl):
                assert_same(ys[l].data.cpu().numpy().reshape(refs[l].packed.shape), refs[l].packed, 256, bits,
                            f"layer {i} level {l}")
            check = torch.full_like(nxt_ws, 0x33)
            aqd.conv_expand_input([(ys[l], None, None, l) for l in range(nl)], Ws[i + 1][0], 1, 1, check)
            torch.cuda.synchronize()
            assert torch.equal(check, nxt_ws), f"chained image of layer {i}"
            cur, cur_ws, nxt_ws = ys, nxt_ws, cur_ws
        cls = wl.convs[4]
        hs = [aqd.DTensor.empty(t.n, t.h, t.w, cls.cout, 32) for t in refs]
        aqd.conv_int_grouped_expanded([(cur[l], hs[l], None, l) for l in range(nl)], Ws[4][0], 1, 1,
                                      rq=aqd.RequantParams.from_numpy(None, None, cls.bias), workspace=cur_ws)
        torch.cuda.synchronize()
        for l in range(nl):
            want = _ref_conv(refs[l], Ws[4][1], cls, level=l).packed
            assert_same(hs[l].data.cpu().numpy().reshape(want.shape), want, cls.cout, 32, f"head level {l}")
    finally:
        aqd.set_conv_path(old)
    assert aqd.device_status() == 0


def test_chain_rejects_overlap_and_bad_shapes():
    rng = np.random.default_rng(5)
    W, _ = weights(synth.weight_codes(rng, (256, 3, 3, 256), 2), 2)
    X = aqd.DTensor.empty(1, 6, 7, 256, 2)
    Y = aqd.DTensor.empty(1, 6, 7, 256, 2)
    jobs = [(X, Y, None, 0)]
    ws = aqd.workspace_for(jobs, W, 1, 1)
    rq = aqd.RequantParams.from_numpy(np.full((1, 256), 1 << 30), np.full((1, 256), 8), np.zeros((1, 256)))
    with pytest.raises(aqd.AqdError) as e:  # output image into the input workspace
        aqd.conv_int_grouped_chain(jobs, W, 1, 1, rq=rq, workspace=ws, next_pad=1, next_workspace=ws)
    assert e.value.status == 1
    small = aqd.workspace_for(jobs, W, 1, 0)  # too small for padding 1
    with pytest.raises(aqd.AqdError) as e:
        aqd.conv_int_grouped_chain(jobs, W, 1, 1, rq=rq, workspace=ws, next_pad=1, next_workspace=small)
    assert e.value.status == 1
    torch.cuda.synchronize()
