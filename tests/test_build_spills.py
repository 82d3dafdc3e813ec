"""The tensor-core kernels that the benchmark step and the head run must compile without
register spills (ptxas reports them by function in the build log): a spill in the tower's
epilogue cost 46% of its time once."""
import os
import re

import pytest

LOG = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "paper_2007_06919_gb300", "_build",
                   "conv_tc.log")

# conv_tc_kernel<kXBits = 2, chunk in tap, workspace path, kPair, no skip, no split, 128-byte chunks, kFp4, kOStage>
HOT = [f"conv_tc_kernelILi2ELb1ELb1ELb{pair}ELb0ELb0ELi128ELb{fp4}ELb{st}E"
       for pair in (0, 1) for fp4 in (0, 1) for st in (0, 1)]


def test_hot_conv_kernels_do_not_spill():
    if not os.path.exists(LOG):
        import __graft_entry__
        __graft_entry__.build()
    if not os.path.exists(LOG):
        pytest.skip("no build log")
    text = open(LOG).read()
    spilled = re.findall(r"spilled to local memory in function '([^']+)'", text)
    bad = [h for h in HOT for f in spilled if h in f]
    assert not bad, f"register spills in {bad}"
