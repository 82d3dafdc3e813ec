"""The whole integer detector of config 3 (integer ResNet-18 + FPN P3-P7 + shared head, 4-bit,
8-bit RGB input) on the GPU against the oracle, every tensor of the network compared.

Reduced sizes are compared whole (every layer output, bit for bit), including a size that
is not a multiple of the network's stride 32 (ragged tiles everywhere, FPN up-reads that
stop short). At the full size (batch 8, 800x1344) every layer output of all eight images is
compared with the oracle's run on the same seeded image codes."""
import numpy as np
import pytest

from paper_2007_06919_gb300 import synth

pytestmark = pytest.mark.gpu


def _gpu_codes(net, name, images=None):
    """The GPU's tensor as int32 codes, unpacked on the CPU by the oracle's unpacker."""
    import oracle
    for f, (a, b, ca) in net.fused.items():
        if name in (a, b):
            full = _gpu_codes(net, f, images)
            return full[..., :ca] if name == a else full[..., ca:]
    t = net.tensors[name]
    raw = t.data.cpu().numpy().reshape(t.n, t.h, t.w, -1)
    n = t.n
    if images is not None:
        raw, n = raw[images], len(images)
    return oracle.CodeTensor(np.ascontiguousarray(raw), n, t.h, t.w, t.c, t.bits).codes()


def _build(batch, h, w, w_pad, **kw):
    import torch
    import oracle
    from paper_2007_06919_gb300.detector import IntDetector
    wl = synth.config3(batch=batch, h=h, w=w, w_pad=w_pad)
    layers = wl.extra["layers"]
    img = oracle.CodeTensor.from_codes(wl.inputs[0], 8)
    net = IntDetector(layers, (batch, h, w_pad, 3, 8), **kw)
    net.tensors["image"].data.copy_(torch.from_numpy(img.packed).reshape(net.tensors["image"].data.shape))
    for k, t in net.tensors.items():
        if k != "image":
            t.data.fill_(0xA5)  # poison: every output byte must be written
    return wl, layers, img, net


@pytest.mark.parametrize("size", [(1, 128, 190, 192), (2, 100, 147, 150)], ids=["128x192", "ragged_100x150"])
@pytest.mark.parametrize("chain,fuse", [(True, True), (False, False)], ids=["fused", "plain"])
def test_detector_reduced_size_bit_exact(size, chain, fuse):
    import torch
    import oracle
    from paper_2007_06919_gb300 import aqd
    wl, layers, img, net = _build(*size, chain=chain, fuse_heads=fuse, fuse_pool=fuse)
    net.forward()
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    ref = oracle.run_network(layers, {"image": img})
    checked = 0
    for ly in layers:
        for d in ly.dst:
            got, want = _gpu_codes(net, d), ref[d].codes()
            assert got.shape == want.shape, d
            bad = np.argwhere(got != want)
            assert bad.size == 0, f"{d}: {len(bad)} mismatches, first at {bad[0].tolist()}"
            checked += 1
    assert checked == sum(len(ly.dst) for ly in layers)
    if chain:
        assert any(p.chain_to is not None for k, p in net.steps if k == "conv")


def test_detector_plan_uses_fast_paths():
    """The planner chains the head tower and fuses the output convs; the bench relies on it.
    Its op count is 2*M*N*K of the unfused convs."""
    from paper_2007_06919_gb300 import aqd
    _, layers, _, net = _build(1, 128, 190, 192)
    chained = [p.layer.name for k, p in net.steps if k == "conv" and p.chain_to is not None]
    for i in range(4):
        assert f"head.tower{i}" in chained
    # the stem's max-pool runs in the first residual stage's expansion pass
    assert not [p for k, p in net.steps if k == "pool"]
    assert [p.pool.name for k, p in net.steps if k == "conv" and p.pool is not None] == ["pool"]
    assert set(net.fused) == {f"cls.{l}+box.{l}" for l in range(5)}
    ops = 0
    for ly in layers:
        if ly.conv is None:
            continue
        cv = ly.conv
        for s in ly.src:
            x = net.tensors[s]
            ho, wo = aqd.conv_out_hw(x.h, x.w, cv.kh, cv.kw, cv.stride, cv.pad)
            ops += 2 * x.n * ho * wo * cv.cout * cv.kh * cv.kw * cv.cin
    assert net.ops == ops


def test_detector_full_size_bit_exact():
    """Batch 8 at 800x1344 on the GPU; every layer output of all eight images against the
    oracle's run of the network (about 1.8 TOP on the host cores)."""
    import torch
    import oracle
    from paper_2007_06919_gb300 import aqd
    wl, layers, img, net = _build(8, 800, 1333, 1344)
    net.forward()
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    ref = oracle.run_network(layers, {"image": img})
    for ly in layers:
        for d in ly.dst:
            got, want = _gpu_codes(net, d), ref[d].codes()
            bad = np.argwhere(got != want)
            assert bad.size == 0, f"{d}: {len(bad)} mismatches, first at {bad[0].tolist()}"
