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
