"""Host logic of bench.py (no GPU): the roofline's traffic comes from the committed ncu
summaries of the workload's model shape, the DRAM bytes of one captured launch against its
algorithmic bytes; the summaries must be parseable and their figures consistent with the
algorithmic bytes the bench computes for the same (rows, context)."""
import subprocess
import sys

import pytest

import bench
import synth


@pytest.mark.parametrize("workload,rows,ctx", [("1.5b", 25, 384), ("3b", 25, 512), ("oversampled", 25, 384)])
def test_traffic_from_the_committed_summaries(workload, rows, ctx):
    got = bench.read_traffic(workload)
    assert got is not None, workload
    traffic, algo = got
    m = synth.WORKLOADS[workload].model
    # the summary's algorithmic bytes are the bench's own formula at the captured (rows, context):
    # weights once (with the norms) + K/V reads of the context + the appends + the embedding rows
    assert algo == bench.step_algorithmic_bytes(m, rows, ctx)
    # written out once more from the model shape, independently of the bench's helpers
    kvtok = m.layers * 2 * m.n_kv_heads * m.head_dim * 2
    assert kvtok == {"1.5b": 28672, "3b": 36864, "oversampled": 28672}[workload]
    # reads equal the algorithmic bytes, the rest are write-backs: a small excess only
    assert algo <= traffic < 1.05 * algo


def test_points_option_is_parsed():
    out = subprocess.run([sys.executable, "bench.py", "--help"], capture_output=True, text=True, cwd=bench.ROOT)
    assert out.returncode == 0 and "--points" in out.stdout
