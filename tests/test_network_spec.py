"""CPU checks of the config-3 network: the seeded layer list (integer ResNet-18 + FPN + head)
is well formed and has the expected size, and the oracle's walk over it applies each layer
as a plain oracle convolution with the right per-level table row."""
import numpy as np
import pytest

from paper_2007_06919_gb300 import synth


def _shape_walk(layers, n, h, w):
    """Output shapes by the conv/pool size formula: name -> (n, h, w, c)."""
    shp = {"image": (n, h, w, 3)}
    for ly in layers:
        for j, (s, d) in enumerate(zip(ly.src, ly.dst)):
            assert s in shp, f"{ly.name} reads {s} before it exists"
            nn, hh, ww, cc = shp[s]
            if ly.pool is not None:
                k, st, p = ly.pool
                cout = cc
            else:
                k, st, p, cout = ly.conv.kh, ly.conv.stride, ly.conv.pad, ly.conv.cout
                assert ly.conv.cin == cc, (ly.name, cc)
            shp[d] = (nn, (hh + 2 * p - k) // st + 1, (ww + 2 * p - k) // st + 1, cout)
            if ly.skip:
                sk = shp[ly.skip[j]]
                up = ly.upsample
                assert sk[3] == cout and sk[1] * up >= shp[d][1] and sk[2] * up >= shp[d][2], ly.name
    return shp


def test_config3_layer_list_is_well_formed():
    wl = synth.config3(batch=1, h=64, w=90, w_pad=96)
    layers = wl.extra["layers"]
    shp = _shape_walk(layers, 1, 64, 96)
    names = [d for ly in layers for d in ly.dst]
    assert len(names) == len(set(names))
    # FPN levels P3..P7 at strides 8..128 of the padded input
    assert [shp[f"P{l}"][1:3] for l in range(3, 8)] == [(8, 12), (4, 6), (2, 3), (1, 2), (1, 1)]
    # 20 backbone convs (conv1 + 16 block convs + 3 downsample), 8 FPN convs, 6 head convs
    assert sum(ly.conv is not None for ly in layers) == 34
    assert sum(ly.pool is not None for ly in layers) == 1
    head = [ly for ly in layers if ly.name.startswith("head.")]
    assert all(len(ly.src) == 5 and ly.conv.m0 is None or ly.conv.m0.shape[0] == 5 for ly in head)
    # the image's padded columns hold code 0
    assert not wl.inputs[0][:, :, 90:].any()


def test_config3_full_size_work():
    """At 800x1344 the levels are the FPN sizes of an 800x1333 image, and the network is
    about 220 GOP per image (1.76 TOP per batch of 8), head tower included."""
    wl = synth.config3(batch=1, h=16, w=16, w_pad=16)  # the layer list does not depend on the size
    layers = wl.extra["layers"]
    shp = _shape_walk(layers, 8, 800, 1344)
    assert [shp[f"P{l}"][1:3] for l in range(3, 8)] == [tuple(x) for x in synth.FPN_LEVELS]
    ops = 0
    for ly in layers:
        if ly.conv is None:
            continue
        for s, d in zip(ly.src, ly.dst):
            n, h, w, c = shp[d]
            ops += 2 * n * h * w * c * ly.conv.kh * ly.conv.kw * ly.conv.cin
    assert 1.6e12 < ops < 1.9e12, ops


def test_config3_is_seeded():
    a = synth.config3(batch=1, h=32, w=30, w_pad=32)
    b = synth.config3(batch=1, h=32, w=30, w_pad=32)
    assert np.array_equal(a.inputs[0], b.inputs[0])
    for x, y in zip(a.convs, b.convs):
        assert np.array_equal(x.w, y.w) and np.array_equal(x.bias, y.bias)


def test_oracle_network_walk(oracle_mod):
    """run_network = one oracle conv per job with table row l for job l, the skip and its
    up-read as listed; outputs stay in their code ranges."""
    oracle = oracle_mod
    wl = synth.config3(batch=1, h=64, w=90, w_pad=96)
    layers = wl.extra["layers"]
    T = oracle.run_network(layers, {"image": oracle.CodeTensor.from_codes(wl.inputs[0], 8)})
    by = {ly.name: ly for ly in layers}
    for ly in layers:
        for d in ly.dst:
            t = T[d]
            if t.bits != 32:
                c = t.codes()
                assert c.min() >= 0 and c.max() <= (1 << t.bits) - 1
    # the head's level-3 job uses row 3 of the per-level tables
    ly = by["head.tower1"]
    cv = ly.conv
    wp = oracle.pack(cv.w.reshape(-1, cv.cin), cv.w_bits)

    def job(level):
        return oracle.conv_int(T[ly.src[3]], wp, cv.w_bits, 0, 3, 3, 1, 1, 256, level=level, m0=cv.m0,
                               shift=cv.shift, bias=cv.bias, levels=5, out_bits=4).packed
    assert np.array_equal(job(3), T[ly.dst[3]].packed)
    assert not np.array_equal(job(0), T[ly.dst[3]].packed)
    # the FPN top-down add reads the coarser map with nearest 2x upsampling
    ly = by["fpn.lat4"]
    cv = ly.conv
    wp = oracle.pack(cv.w.reshape(-1, cv.cin), cv.w_bits)
    got = oracle.conv_int(T[ly.src[0]], wp, 4, 0, 1, 1, 1, 0, 256, m0=cv.m0, shift=cv.shift, bias=cv.bias,
                          skip=T["fpn.m5"], skip_c=cv.skip_c, skip_d=cv.skip_d, upsample=2, out_bits=4)
    assert np.array_equal(got.packed, T["fpn.m4"].packed)
    # and the skip is visible: without it the output differs
    plain = oracle.conv_int(T[ly.src[0]], wp, 4, 0, 1, 1, 1, 0, 256, m0=cv.m0, shift=cv.shift, bias=cv.bias,
                            out_bits=4)
    assert not np.array_equal(plain.packed, T["fpn.m4"].packed)
    # the downsample branch enters the next conv as an int32 skip
    assert T["layer3.0.down"].bits == 32 and by["layer3.0.conv_b"].skip == ["layer3.0.down"]
