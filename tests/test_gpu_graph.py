"""The convolution replayed from CUDA graphs, as the benchmark runs it: a tower layer
(256->256, 2-bit) and the fused 256->84 int32 output conv captured in one graph, a second
graph with only the tower layer captured after it, then the first graph replayed; every
output must equal the oracle's. (The two convs have different shared-memory plans, so
this also checks that a later capture leaves an earlier graph launchable.)"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_same, to_device, weights
from paper_2007_06919_gb300 import aqd, synth

pytestmark = pytest.mark.gpu


def test_graph_replay_after_later_capture_bit_exact():
    levels = [(12, 21), (6, 11)]
    wl = synth.head_tower(21, 2, 2, levels=levels, calibrated=True)
    tower, cls, box = wl.convs[0], wl.convs[4], wl.convs[5]
    xts = [oracle.CodeTensor.from_codes(x, 2) for x in wl.inputs]
    Wt, wpt = weights(tower.w, 2)
    Wh, _ = weights(np.concatenate([cls.w, box.w]), 2)
    rq_t = aqd.RequantParams.from_numpy(tower.m0, tower.shift, tower.bias)
    rq_h = aqd.RequantParams.from_numpy(None, None, np.concatenate([cls.bias, box.bias], axis=1))
    xs = [to_device(t) for t in xts]
    mid = [aqd.DTensor.empty(t.n, t.h, t.w, 256, 2) for t in xts]
    out = [aqd.DTensor.empty(t.n, t.h, t.w, 84, 32) for t in xts]
    jobs_t = [(xs[l], mid[l], None, l) for l in range(2)]
    jobs_h = [(mid[l], out[l], None, l) for l in range(2)]
    ws = aqd.workspace_for(jobs_t, Wt, 1, 1)
    stream = torch.cuda.Stream()
    torch.cuda.synchronize()
    g1, g2 = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g1, stream=stream):
        aqd.conv_int_grouped(jobs_t, Wt, 1, 1, rq=rq_t, workspace=ws, stream=stream)
        aqd.conv_int_grouped(jobs_h, Wh, 1, 1, rq=rq_h, workspace=ws, stream=stream)
    with torch.cuda.graph(g2, stream=stream):
        aqd.conv_int_grouped(jobs_t, Wt, 1, 1, rq=rq_t, workspace=ws, stream=stream)
    for t in mid + out:
        t.data.fill_(0xA5)
    torch.cuda.synchronize()
    g1.replay()
    torch.cuda.synchronize()
    assert aqd.device_status() == 0
    for l in range(2):
        r_mid = oracle.conv_int(xts[l], wpt, 2, 0, 3, 3, 1, 1, 256, level=l, m0=tower.m0, shift=tower.shift,
                                bias=tower.bias, levels=2, out_bits=2)
        assert_same(mid[l].data.cpu().numpy().reshape(r_mid.packed.shape), r_mid.packed, 256, 2, f"tower {l}")
        got = out[l].data.cpu().numpy().view(np.int32).reshape(-1, 84)
        for cv, lo in ((cls, 0), (box, 80)):
            wp = oracle.pack(cv.w.reshape(-1, cv.cin), 2)
            want = oracle.conv_int(r_mid, wp, 2, 0, 3, 3, 1, 1, cv.cout, level=l, bias=cv.bias, levels=2,
                                   out_bits=32).packed.view(np.int32).reshape(-1, cv.cout)
            assert np.array_equal(got[:, lo:lo + cv.cout], want), f"head {cv.cout} level {l}"
