"""Host-side logic of bench.py: byte accounting, clock parsing, rank aggregation (CPU)."""

import os
import socket

import pytest
import torch
import torch.multiprocessing as mp

import bench
from paper_2609_30656_gb300 import metrics, workloads as wl


def test_forward_and_backward_bytes_by_hand():
    # 2 tables (dims 4 and 8, fp16), batch 3, lookups 5 and 2.
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts((4, 8), 2, 3, off, weighted=True)
    assert c.lookups_per_table == (5, 2) and c.n == 7 and c.sum_dims == 12
    f = metrics.forward_bytes(c)
    assert f["rows"] == 5 * 4 * 2 + 2 * 8 * 2
    assert f["indices"] == 7 * 8 and f["offsets"] == 7 * 8 and f["weights"] == 7 * 4
    assert f["output"] == 3 * 12 * 4
    assert f["total"] == sum(v for k, v in f.items() if k != "total")
    b = metrics.backward_bytes(c, [3, 1])
    assert b["grad_gather"] == 5 * 4 * 4 + 2 * 8 * 4
    assert b["unique_ids"] == 4 * 8 and b["grads"] == 3 * 4 * 4 + 1 * 8 * 4
    assert metrics.forward_unique_bytes(c, [3, 1]) == f["total"] - f["rows"] + 3 * 8 + 1 * 16


def test_compulsory_bytes_by_hand():
    # 2 tables (dims 4 and 8, fp16), batch 3: table 0 has bags of 2, 0, 3 lookups,
    # table 1 bags of 1, 1, 0 -> 2 and 2 non-empty bags; 3 and 1 distinct rows
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts((4, 8), 2, 3, off, weighted=False)
    assert c.nonempty_per_table == (2, 2)
    cb = metrics.component_compulsory_bytes(c, [3, 1], packed=False)
    assert cb["fwd.gather"] == metrics.forward_unique_bytes(c, [3, 1])
    slices = 2 * 4 * 4 + 2 * 8 * 4
    grads = 3 * 4 * 4 + 1 * 8 * 4
    assert cb["bwd.reduce"] == slices + 4 * 7 + 4 * 4 + grads + 16 * 4
    assert metrics.component_compulsory_bytes(c, [3, 1], packed=True)["bwd.reduce"] == cb["bwd.reduce"] + 8 * 7


def test_weight_grad_bytes_by_hand():
    # 2 tables (dims 4 and 8, fp16), batch 3, lookups 5 and 2
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts((4, 8), 2, 3, off, weighted=False)
    rows = 5 * 4 * 2 + 2 * 8 * 2
    slices = 5 * 4 * 4 + 2 * 8 * 4
    assert metrics.weight_grad_bytes(c) == rows + slices + 7 * (8 + 4) + 7 * 8


def test_apply_step_bytes_by_hand():
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts((4, 8), 2, 3, off, weighted=False)
    b = metrics.backward_bytes(c, [3, 1])
    rows = 3 * 4 * 2 + 1 * 8 * 2
    assert metrics.apply_step_bytes(c, [3, 1], False) == b["total"] - b["grads"] - b["unique_ids"] + 2 * rows
    assert metrics.apply_step_bytes(c, [3, 1], True) == metrics.apply_step_bytes(c, [3, 1], False) + 4 * 8


def test_sparse_apply_bytes_by_hand():
    # 3 touched rows of the dim-4 fp16 table, 1 of the dim-8 one
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts((4, 8), 2, 3, off, weighted=False)
    ids = 4 * 16
    grads = (3 * 4 + 8) * 4
    rows = 2 * (3 * 4 + 8) * 2
    assert metrics.sparse_apply_bytes(c, [3, 1], False) == ids + grads + rows
    assert metrics.sparse_apply_bytes(c, [3, 1], True) == ids + grads + rows + 4 * 8


def test_fm_bytes_by_hand():
    # 3 samples x 2 fields x dim 4: 24 floats of pooled rows
    assert metrics.fm_bytes(3, 2, 4, backward=False) == 24 * 4 + 3 * 4
    assert metrics.fm_bytes(3, 2, 4, backward=True) == 2 * 24 * 4 + 3 * 4


def test_radix_passes_follow_row_bits():
    # keys 0 .. rows_t (the spare key rows_t marks an out-of-range lookup)
    assert metrics.radix_passes([255]) == 1
    assert metrics.radix_passes([256]) == 2
    assert metrics.radix_passes([257]) == 2
    assert metrics.radix_passes([5_000_000] * 100) == 3   # 23-bit rows, per-table ranges
    assert metrics.radix_passes([100_000] * 8) == 3       # 17-bit rows
    assert metrics.radix_passes([1000, 70000]) == 3       # the largest table decides
    assert metrics.sort_bytes(10, 3) == 480


def test_workload_description_names_the_shape():
    d = bench.describe(wl.get_workload("cfg5"))
    assert "100 x 5,000,000 rows" in d and "batch 65536" in d and "Zipf(1.2)" in d
    assert "5% empty" in d and "sum pooling" in d
    assert "weighted mean" in bench.describe(wl.get_workload("cfg4"))


def test_clock_summary_parsing():
    s = bench.ClockSampler(0)
    s.out = ("1965, 2070, 900.5, Not Active, Not Active, Not Active, Active\n"
             "1980, 2070, 950.0, Not Active, Not Active, Not Active, Not Active\n"
             "300, 2070, 80.0, Not Active, Not Active, Not Active, Not Active\n")
    r = s.summary()
    assert r["sm_max_mhz"] == 2070 and r["sm_mhz"] == pytest.approx(1972.5)
    assert r["reasons"] == ["sw_power_cap"]
    s.out = ""
    assert s.summary()["reasons"] == ["unsampled"]


def test_traffic_is_null_unless_recorded_for_this_source(tmp_path, monkeypatch):
    assert bench.recorded_traffic("fwd.gather", "no-such-workload") is None
    assert len(bench.kernel_source_hash()) == 16
    for k in bench.KERNEL_SOURCES:  # every listed source exists
        assert len(bench.kernel_source_hash(k)) == 16


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    # rank r took (r + 1) ms and moved (r + 1) GB
    res = bench.aggregate(float(rank + 1), 1e9 * (rank + 1), 100.0 * (rank + 1), world)
    q.put((rank, res))
    torch.distributed.destroy_process_group()


def test_aggregate_takes_max_time_and_summed_work_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        ms, nbytes, rows = got[r]
        assert ms == 2.0 and nbytes == 3e9 and rows == 300.0


def test_aggregate_is_identity_on_one_rank():
    assert bench.aggregate(1.5, 2.0, 3.0, 1) == (1.5, 2.0, 3.0)


def test_report_written_from_measured_components(tmp_path):
    import json
    w = wl.scaled(wl.get_workload("cfg5"), num_tables=2, batch=3, rows=10)
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts(w.dims, w.elem_bytes, w.batch, off, weighted=False)
    comp_ms = {"fwd.prep": 0.01, "fwd.gather": 1.0, "fwd.fixup": 0.01, "bwd.keygen": 0.2,
               "bwd.sort": 0.5, "bwd.rle": 0.1, "bwd.reduce": 2.0}
    comp_bytes = {"fwd.gather": 6e9, "bwd.reduce": 8e9}  # per step (the breakdown run's mean)
    line = {"steps": 3, "ms_per_step": 4.0, "config": {"workload": "tiny"},
            "next_rows": {"fm": {"forward": {"ms": 0.1, "bytes": 1e6}, "backward": {"ms": 0.2, "bytes": 2e6}},
                          "weight_grad": {"ms": 0.3, "bytes": 3e6},
                          "backward_apply": {"sgd": {"ms": 3.0, "bytes": 4e6}}}}
    bench.write_report(str(tmp_path / "r"), w, line, comp_ms, comp_bytes, [c], [[3, 1]], 1000.0)
    doc = json.loads((tmp_path / "r.json").read_text())
    names = [r["component"] for r in doc["components"]]
    assert names[:4] == ["run", "run/step", "run/step/forward", "run/step/forward/fwd.prep"]
    assert "run/next/fm.forward" in names and "run/next/backward_apply.sgd" in names
    gather = doc["components"][names.index("run/step/forward/fwd.gather")]
    assert gather["est_avg_bw_gbs"] == pytest.approx(6000.0)  # 6 GB in 1 ms
    bwd = doc["components"][names.index("run/step/backward")]
    assert bwd["latency_ms"] == pytest.approx(2.8) and bwd["est_avg_bw_gbs"] == pytest.approx(8e9 / 2.8e-3 / 1e9, abs=0.1)
    step = doc["components"][names.index("run/step")]
    assert step["latency_ms"] == 4.0 and step["measured"]
    # the step's rate covers its own kernels: (6 + 8) GB over their 3.82 ms
    assert step["est_avg_bw_gbs"] == pytest.approx(14e9 / 3.82e-3 / 1e9, abs=0.1)
    assert "| fwd.gather |" in (tmp_path / "r.md").read_text().replace("&nbsp;", "")


def test_quantiles_and_timing_summary():
    xs = [5.0, 1.0, 3.0, 2.0, 4.0]
    assert bench.quantile(xs, 0.5) == 3.0
    assert bench.quantile(xs, 0.1) == pytest.approx(1.4)
    assert bench.quantile(xs, 0.9) == pytest.approx(4.6)
    s = bench.timing_summary(xs)
    assert s["median"] == 3.0 and s["p10"] == 1.4 and s["p90"] == 4.6 and s["samples"] == 5


def test_roofline_uses_dram_traffic_when_recorded(monkeypatch):
    w = wl.scaled(wl.get_workload("cfg5"), num_tables=2, batch=3, rows=10)
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts(w.dims, w.elem_bytes, w.batch, off, weighted=False)
    comp_ms = {"fwd.gather": 1.0, "bwd.reduce": 2.0}
    comp_bytes = {"fwd.gather": 6e9, "bwd.reduce": 40e9}  # 20 TB/s of every-lookup bytes
    comp_compulsory = {"fwd.gather": 1e9, "bwd.reduce": 4e9}
    monkeypatch.setattr(bench, "recorded_traffic", lambda k, wl_: None)
    r = bench.roofline_of("x", comp_ms, comp_bytes, comp_compulsory, 5000.0, "measured", None, [c], w)
    assert r["kernel"] == "bwd.reduce" and r["basis"] == "compulsory"
    assert r["achieved"] == pytest.approx(2000.0) and r["frac"] == pytest.approx(0.4)
    assert r["alg_frac"] == pytest.approx(4.0)  # the reuse-inflated figure under its own name
    monkeypatch.setattr(bench, "recorded_traffic", lambda k, wl_: 6e9)
    r = bench.roofline_of("x", comp_ms, comp_bytes, comp_compulsory, 5000.0, "measured", None, [c], w)
    assert r["basis"] == "dram" and r["frac"] == pytest.approx(0.6) and r["traffic"] == 6e9
    ceiling = {"512": {"gbs": 20000.0}, "256": {"gbs": 20000.0}}
    r = bench.roofline_of("x", comp_ms, comp_bytes, comp_compulsory, 5000.0, "measured", ceiling, [c], w)
    gathered = metrics.backward_bytes(c, [0, 0])["grad_gather"]
    assert r["l2_gather_gbs"] == round(gathered / 2e-3 / 1e9, 1)
    assert r["frac_l2"] == pytest.approx(gathered / 2e-3 / 1e9 / 20000.0, abs=1e-4)
    assert r["l2_ceiling_row_bytes"] == 512  # fp32 grad_out slices of dim 128


def test_forward_gather_against_both_l2_rates():
    # fp16 rows of dim 128 (256 bytes): against the plain gather rate and the
    # rate with the forward's widening adds
    w = wl.scaled(wl.get_workload("cfg5"), num_tables=2, batch=3, rows=10)
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts(w.dims, w.elem_bytes, w.batch, off, weighted=False)
    rows = 7 * 128 * 2  # 7 lookups of 256-byte rows
    assert metrics.forward_bytes(c)["rows"] == rows
    ceiling = {"256": {"gbs": 20000.0, "f16_sum_gbs": 16000.0}}
    r = bench.gather_vs_l2(1e-6, [c], w, ceiling)  # 1 ns
    assert r["l2_gather_gbs"] == round(rows / 1e-9 / 1e9, 1) and r["l2_ceiling_row_bytes"] == 256
    assert r["frac_l2"] == pytest.approx(rows / 1e-9 / 1e9 / 20000.0, abs=1e-4)
    assert r["frac_l2_widened"] == pytest.approx(rows / 1e-9 / 1e9 / 16000.0, abs=1e-4)
    assert bench.gather_vs_l2(1e-6, [c], w, {"512": {"gbs": 1.0}}) == {}


def test_roofline_of_a_streaming_kernel_uses_its_algorithmic_bytes(monkeypatch):
    # the sort can be the longest component (e.g. with serialised launches); it has
    # no reuse, so its algorithmic bytes are its compulsory ones
    w = wl.scaled(wl.get_workload("cfg5"), num_tables=2, batch=3, rows=10)
    off = torch.tensor([0, 2, 2, 5, 6, 7, 7])
    c = metrics.batch_counts(w.dims, w.elem_bytes, w.batch, off, weighted=False)
    monkeypatch.setattr(bench, "recorded_traffic", lambda k, wl_: None)
    r = bench.roofline_of("x", {"bwd.sort": 3.0, "bwd.reduce": 1.0}, {"bwd.sort": 9e9, "bwd.reduce": 1e9},
                          {"bwd.reduce": 1e8}, 5000.0, "measured", None, [c], w)
    assert r["kernel"] == "bwd.sort" and r["basis"] == "algorithmic" and r["frac"] == pytest.approx(0.6)
