"""Per-layer code histograms of the calibrated synthetic workloads, computed with the CPU
oracle and printed (pytest -s shows them). The workloads' requant is drawn around the shift
that spreads the accumulator's standard deviation over the code range, so every layer's
codes must stay spread: all 2^k codes present, the ReLU clip at 0 near half of the outputs,
and the clip at the top code a minority. A recipe that drove a layer's codes all to 0 or
all to the top (as config 1's literal shifts would through 34 layers) fails here."""
import numpy as np

from paper_2007_06919_gb300 import synth


def _hist(t):
    c = t.codes()
    return np.bincount(c.ravel(), minlength=1 << t.bits) / c.size


def test_config3_codes_stay_spread_in_every_layer(oracle_mod):
    oracle = oracle_mod
    wl = synth.config3(batch=1, h=128, w=180, w_pad=192)
    layers = wl.extra["layers"]
    T = oracle.run_network(layers, {"image": oracle.CodeTensor.from_codes(wl.inputs[0], 8)})
    rows = []
    for ly in layers:
        for d in ly.dst:
            t = T[d]
            if t.bits == 32:
                continue
            h = _hist(t)
            rows.append((d, h))
            assert (h > 0).all(), f"{d}: codes missing {np.flatnonzero(h == 0).tolist()}"
            assert 0.2 <= h[0] <= 0.7, f"{d}: {h[0]:.2f} of the codes are 0"
            assert h[-1] <= 0.35, f"{d}: {h[-1]:.2f} of the codes are at the top"
    print("\nconfig 3 (batch 1, 128 x 192): layer, share of code 0, share of code 15, histogram")
    for d, h in rows:
        print(f"  {d:14s} {h[0]:.2f} {h[-1]:.3f} " + " ".join(f"{v:.3f}" for v in h))
    assert len(rows) == 46  # conv1, the pool, 16 backbone convs, 3 laterals, P3-P7, 20 head convs


def test_calibrated_head_tower_codes(oracle_mod):
    oracle = oracle_mod
    levels = [(25, 42), (13, 21)]
    wl = synth.head_tower(2, 1, 2, levels=levels, calibrated=True)
    xs = [oracle.CodeTensor.from_codes(v, 2) for v in wl.inputs]
    print("\ncalibrated 2-bit head tower (batch 1, levels 25x42 and 13x21): layer, level, histogram")
    for i, cv in enumerate(wl.convs[:4]):
        wp = oracle.pack(cv.w.reshape(-1, cv.cin), cv.w_bits)
        xs = [oracle.conv_int(x, wp, 2, 0, 3, 3, 1, 1, 256, level=lv, m0=cv.m0, shift=cv.shift, bias=cv.bias,
                              levels=len(levels), out_bits=2) for lv, x in enumerate(xs)]
        for lv, x in enumerate(xs):
            h = _hist(x)
            print(f"  tower {i} level {lv}: " + " ".join(f"{v:.3f}" for v in h))
            assert (h > 0.03).all() and h[0] <= 0.75 and h[-1] <= 0.2
