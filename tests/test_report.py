"""The component report's aggregation rules (CPU): a parent without its own
latency sums its children; its rates are latency-weighted means over the
measured leaves, i.e. total bytes (FLOPs) over total leaf latency."""

import json

import pytest

from paper_2609_30656_gb300 import metrics, report
from paper_2609_30656_gb300.report import Component


def _tree():
    root = Component("step")
    a = root.add(Component("a"))
    a.add(Component("a1", 2.0, bytes=2e9, flops=1e9))      # 1000 GB/s, 0.5 TFLOP/s
    a.add(Component("a2", 6.0, bytes=12e9, flops=0.0))     # 2000 GB/s, 0
    root.add(Component("b", 2.0, bytes=1e9, flops=4e9))    # 500 GB/s, 2 TFLOP/s
    return root


def test_parent_latency_is_the_sum_and_rates_are_latency_weighted():
    root = _tree()
    a = root.children[0]
    assert report.latency(a) == 8.0 and report.latency(root) == 10.0
    # (1000 * 2 + 2000 * 6) / 8 = 1750 GB/s = 14 GB / 8 ms
    assert report.bandwidth_gbs(a) == pytest.approx(1750.0)
    assert report.bandwidth_gbs(root) == pytest.approx(15e9 / 10e-3 / 1e9)
    assert report.tflops(root) == pytest.approx(5e9 / 10e-3 / 1e12)


def test_a_measured_parent_keeps_its_latency():
    root = _tree()
    root.latency_ms = 11.0  # gaps between kernels
    assert report.latency(root) == 11.0
    assert report.bandwidth_gbs(root) == pytest.approx(1500.0)  # still from the leaves


def test_rows_json_and_markdown():
    rows = report.rows(_tree(), peak_gbs=2000.0, peak_tflops=10.0)
    assert [r["component"] for r in rows] == ["step", "step/a", "step/a/a1", "step/a/a2", "step/b"]
    assert [r["depth"] for r in rows] == [0, 1, 2, 2, 1]
    a1 = rows[2]
    assert a1["bw_util_pct"] == 50.0 and a1["mfu_pct"] == 5.0 and a1["measured"]
    assert not rows[1]["measured"]
    doc = json.loads(report.to_json(_tree(), 2000.0, 10.0, workload="w"))
    assert doc["workload"] == "w" and len(doc["components"]) == 5
    md = report.to_markdown(_tree(), 2000.0, 10.0, title="t")
    assert "| a1 |" in md.replace("&nbsp;", "") and "(sum)" in md


def test_step_tree_from_component_timings():
    ms = {"fwd.prep": 0.1, "fwd.gather": 6.0, "fwd.fixup": 0.01, "bwd.keygen": 1.0,
          "bwd.sort": 4.0, "bwd.rle": 0.4, "bwd.reduce": 8.0}
    t = report.step_tree(ms, {"fwd.gather": 6e9}, {}, table_mb=100.0, workspace_mb=10.0,
                         extra={"fm.forward": (0.5, 3e9, 1e9)})
    assert [c.name for c in t.children] == ["step", "next"]
    step = t.children[0]
    assert [c.name for c in step.children] == ["forward", "backward"]
    assert [c.name for c in step.children[0].children] == ["fwd.prep", "fwd.gather", "fwd.fixup"]
    assert report.latency(step.children[1]) == pytest.approx(13.4)
    assert step.size_mb == 110.0
    # the step's rates come from its own kernels only, not from the rows beside it
    assert report.bandwidth_gbs(step) == pytest.approx(6e9 / (sum(ms.values()) * 1e-3) / 1e9)


def test_component_flops_by_hand():
    import torch
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts((4, 8), 2, 3, off, weighted=False)
    f = metrics.component_flops(c, [3, 1], mean=False)
    assert f["fwd.gather"] == 5 * 4 + 2 * 8 and f["bwd.reduce"] == 5 * 4 + 2 * 8
    fm = metrics.component_flops(c, [3, 1], mean=True)
    assert fm["fwd.gather"] == 2 * (5 * 4 + 2 * 8) + 3 * 12
    assert f["bwd.sort"] == 0
