"""Host-side pieces of bench.py that need no GPU: the oracle timing of configs 0 and 1 that
the sweep reports beside the GPU numbers (all host cores and one core)."""
import bench


def test_oracle_config_timing_counts_the_config_work():
    ops, secs = bench.oracle_config_timing("config0", 1)
    assert ops == 2 * 32 * 32 * 64 * 64 * 9   # 3x3 64->64 on 32x32, batch 1
    assert secs > 0
    ops, secs = bench.oracle_config_timing("config1", bench.omp_threads())
    m = 2 * 100 * 152
    assert ops == 2 * m * (512 * 128 + 128 * 128 * 9 + 128 * 512)


def test_reference_arm_prints_the_contract_line():
    """`bench.py --impl reference` (the oracle on the host cores, no GPU) prints one JSON line
    with the contract's keys, on the same metric and workload as the GPU arm."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0"],
                       cwd=root, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in line, k
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC and line["unit"] == "TOPS"
    assert line["value"] > 0 and line["higher_is_better"] is True and line["vs_baseline"] is None
    assert line["config"]["workload"] == bench.WORKLOAD
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": "TOPS", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
