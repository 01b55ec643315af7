"""Hierarchical component report of the library's own step, after Component Benchmark.

The paper's result table (Sec. IV.B.1) lists every submodule under its
hierarchical path with its latency, static memory, TFLOP/s, MFU and estimated
bandwidth / bandwidth utilisation; a "container" module with no measurement of
its own takes, for its rates, the latency-weighted mean over its measured
leaves (Sec. IV.A.2 on inter_arch.deep_fm.dense_module), and a parent that could
not be profiled is estimated from its children (Sec. III, recursive profiling).

Here the components are the library's kernels grouped by direction
(``run / step / forward / fwd.gather`` ...). A leaf carries a measured latency and its
algorithmic bytes and FLOPs; a parent without a latency of its own gets the sum
of its children's (the kernels run one after another on one stream). Rates of a
parent are latency-weighted means of its leaves' rates, which equal its total
bytes (or FLOPs) over its total latency.
"""

from __future__ import annotations

import json
from dataclasses import dataclass, field


@dataclass
class Component:
    name: str
    latency_ms: float | None = None   # measured; None = estimated from the children
    bytes: float = 0.0                # algorithmic bytes moved (leaves)
    flops: float = 0.0                # algorithmic floating-point operations (leaves)
    size_mb: float | None = None      # static memory footprint
    children: list["Component"] = field(default_factory=list)

    def add(self, child: "Component") -> "Component":
        self.children.append(child)
        return child


def leaves(c: Component) -> list[Component]:
    return [c] if not c.children else [x for ch in c.children for x in leaves(ch)]


def latency(c: Component) -> float:
    """Measured latency, or the sum over the children when the node has none."""
    if c.latency_ms is not None:
        return c.latency_ms
    return sum(latency(ch) for ch in c.children)


def weighted_rate(c: Component, rate) -> float:
    """Latency-weighted mean of `rate(leaf)` over the measured leaves of c."""
    ls = [x for x in leaves(c) if x.latency_ms]
    tot = sum(x.latency_ms for x in ls)
    return sum(rate(x) * x.latency_ms for x in ls) / tot if tot > 0 else 0.0


def bandwidth_gbs(c: Component) -> float:
    if not c.children:
        return c.bytes / (c.latency_ms * 1e-3) / 1e9 if c.latency_ms else 0.0
    return weighted_rate(c, bandwidth_gbs)


def tflops(c: Component) -> float:
    if not c.children:
        return c.flops / (c.latency_ms * 1e-3) / 1e12 if c.latency_ms else 0.0
    return weighted_rate(c, tflops)


def rows(root: Component, peak_gbs: float, peak_tflops: float) -> list[dict]:
    """One row per component, depth-first, with the paper's result-table columns."""
    out = []

    def walk(c: Component, path: str, depth: int):
        p = f"{path}/{c.name}" if path else c.name
        bw = bandwidth_gbs(c)
        tf = tflops(c)
        out.append({
            "component": p, "depth": depth,
            "latency_ms": round(latency(c), 4),
            "measured": c.latency_ms is not None,
            "size_mb": None if c.size_mb is None else round(c.size_mb, 1),
            "est_avg_bw_gbs": round(bw, 1),
            "bw_util_pct": round(100 * bw / peak_gbs, 2) if peak_gbs else None,
            "tflops": round(tf, 4),
            "mfu_pct": round(100 * tf / peak_tflops, 4) if peak_tflops else None,
        })
        for ch in c.children:
            walk(ch, p, depth + 1)

    walk(root, "", 0)
    return out


def to_json(root: Component, peak_gbs: float, peak_tflops: float, **meta) -> str:
    return json.dumps({"peaks": {"hbm_gbs": peak_gbs, "tflops": peak_tflops}, **meta,
                       "components": rows(root, peak_gbs, peak_tflops)}, indent=1)


def to_markdown(root: Component, peak_gbs: float, peak_tflops: float, title: str = "") -> str:
    head = [f"# {title}", ""] if title else []
    lines = head + [
        "| component | latency (ms) | size (MB) | est. avg BW (GB/s) | BW util | TFLOP/s | MFU |",
        "|---|---:|---:|---:|---:|---:|---:|"]
    for r in rows(root, peak_gbs, peak_tflops):
        name = "&nbsp;&nbsp;" * r["depth"] + r["component"].rsplit("/", 1)[-1]
        lat = f"{r['latency_ms']:.3f}" + ("" if r["measured"] else " (sum)")
        size = "" if r["size_mb"] is None else f"{r['size_mb']:.1f}"
        util = "" if r["bw_util_pct"] is None else f"{r['bw_util_pct']:.1f} %"
        mfu = "" if r["mfu_pct"] is None else f"{r['mfu_pct']:.3f} %"
        lines.append(f"| {name} | {lat} | {size} | {r['est_avg_bw_gbs']:.0f} | {util} | "
                     f"{r['tflops']:.3f} | {mfu} |")
    lines += ["", "Parents without a latency of their own show the sum of their children; their "
              "rates are latency-weighted means over the measured leaves."]
    return "\n".join(lines) + "\n"


def step_tree(comp_ms: dict[str, float], comp_bytes: dict[str, float], comp_flops: dict[str, float],
              table_mb: float, workspace_mb: float, extra: dict[str, tuple[float, float, float]] | None = None
              ) -> Component:
    """The run's tree from per-component latency, bytes and FLOPs: ``run / step /
    {forward, backward} / <kernels>``, and beside the step ``run / next / <extra>``
    for the further rows timed on their own (name -> (ms, bytes, flops))."""
    root = Component("run")
    step = root.add(Component("step", size_mb=table_mb + workspace_mb))
    for direction, prefix in (("forward", "fwd."), ("backward", "bwd.")):
        node = step.add(Component(direction, size_mb=table_mb))
        for name in comp_ms:
            if name.startswith(prefix):
                node.add(Component(name, comp_ms[name], comp_bytes.get(name, 0.0),
                                   comp_flops.get(name, 0.0)))
    if extra:
        nxt = root.add(Component("next"))
        for name, (ms, b, f) in extra.items():
            nxt.add(Component(name, ms, b, f))
    return root
