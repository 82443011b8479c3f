"""Host-side checks of the verification kernel's share split (no GPU).

`CostPartition` in csrc/common.cuh splits the tile sequence of a
tree_verify_attn call into one share per CTA so that every share costs the
same, a switch from one (sequence, cached head) slab to the next counted as w
tiles.  Its arithmetic is plain integer code shared by host and device, so
tests/partition_check.cu compiles the library's own header for the host and
checks it on seeded random batches: the shares cover the tile sequence exactly
and in order, the merge bookkeeping's lookup of any tile names the share that
holds it, and no share costs more than its part of the cost line.
"""
import os
import subprocess
import tempfile

from paper_2402_02082_gb300 import build

HERE = os.path.dirname(os.path.abspath(__file__))


def test_cost_partition_host_check():
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "partition_check")
        cmd = [build.nvcc(), *build.ARCH, "-std=c++17", "-O2", "--expt-relaxed-constexpr",
               "-I", build.CSRC, "-I", build.INCLUDE, os.path.join(HERE, "partition_check.cu"), "-o", exe]
        r = subprocess.run(cmd, capture_output=True, text=True)
        assert r.returncode == 0, r.stdout + r.stderr
        r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
        assert r.returncode == 0 and r.stdout.startswith("ok"), r.stdout + r.stderr
