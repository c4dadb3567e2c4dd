"""bench.py's host-side bookkeeping, on CPU: the DRAM-traffic figure of the
roofline field is read from the committed ncu table only for the workload it
was captured on, and the algorithmic byte counts of the gather modes add up.
"""
import os

import bench
from paper_2608_24063_gb300 import synth
from paper_2608_24063_gb300 import viscache as vc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rows():
    out = []
    for line in open(os.path.join(ROOT, "profiles", "traffic.md")):
        cells = [c.strip() for c in line.strip().strip("|").split("|")]
        if len(cells) == 5 and cells[4].isdigit():
            out.append(cells)
    return out


def test_traffic_table_names_workload_source_and_digest():
    rows = _rows()
    assert {r[0] for r in rows} >= {"score_lse_tc", "score_colsum_tc", "fuse_v_tc", "decode_attn"}
    for kernel, workload, src, digest, nbytes in rows:
        assert workload, kernel
        assert os.path.exists(os.path.join(ROOT, src)), src
        assert len(digest) == 16 and int(digest, 16) >= 0
        assert int(nbytes) > 0


def test_traffic_only_for_the_captured_workload():
    for kernel, workload, _, _, _ in _rows():
        assert bench.traffic_for(kernel, None) is None
        assert bench.traffic_for(kernel, workload + " (other)") is None
    assert bench.traffic_for("no_such_kernel", "workload 3") is None


def test_gather_byte_counts():
    wl = synth.WORKLOADS[3]
    plans = bench.plans_for(wl, vc)
    w = bench.algorithmic(wl, plans)
    assert w["gather_kv_bytes"] == w["gather_bytes"] + w["gather_v_bytes"]
    assert w["gather_v_bytes"] == 2 * w["surv_v_bytes"]
