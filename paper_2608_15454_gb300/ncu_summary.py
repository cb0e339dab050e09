"""Summarise an Nsight Compute launch list of the eager decode step.

Input: the CSV that `ncu --metrics gpu__time_duration.sum[,dram__bytes_read.sum,
dram__bytes_write.sum] --csv --log-file launches.csv python bench.py --eager ...` writes.
Output (markdown on stdout): per kernel, the launches, device time and share of one decode
step, averaged over the complete steps of the capture (a step starts at its first planning
kernel); with the DRAM metrics, the DRAM bytes per launch of the linear-layer and attention
kernel families. `--traffic FILE` merges those per-launch bytes into FILE (JSON), keyed by
workload and family and tagged with the SHA-256 of the family's CUDA sources, so that a reader
can tell when the counters no longer describe the kernels.

    python -m paper_2608_15454_gb300.ncu_summary launches.csv --workload paper_b1 \\
        [--traffic profiles/traffic.json]
"""
from __future__ import annotations

import argparse
import collections
import csv
import hashlib
import json
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
KERNEL_SOURCES = {"linear": ["paper_2608_15454_gb300/csrc/kernels_linear.cu",
                             "paper_2608_15454_gb300/csrc/kernels_umma.cu",
                             "paper_2608_15454_gb300/csrc/epilogue.cuh"],
                  "attention": ["paper_2608_15454_gb300/csrc/kernels_attn.cu"]}
FAMILY = {"linear": ("k_gemv", "k_tgemm", "k_umma", "k_split_rows", "k_gemm", "k_rowstats"),
          "attention": ("k_attn",)}
STEP_MARKERS = ("k_mb_plan", "k_mlp_plan")


def source_hash(kind: str) -> str:
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kind]:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def load(path):
    """Launches in order: (kernel name, grid, block, {metric: value})."""
    launches = collections.OrderedDict()
    hdr = None
    with open(path) as f:
        for r in csv.reader(f):
            if r and r[0] == "ID":
                hdr = r
                continue
            if not hdr or len(r) != len(hdr):
                continue
            d = dict(zip(hdr, r))
            name = re.sub(r"lca::<unnamed>::|lca::|\(anonymous namespace\)::|void ", "", d["Kernel Name"])
            name = re.sub(r"\(.*", "", name).strip()
            e = launches.setdefault(d["ID"], [name, d["Grid Size"], d["Block Size"], {}])
            v = float(d["Metric Value"].replace(",", ""))
            unit = d["Metric Unit"]
            if d["Metric Name"] == "gpu__time_duration.sum":
                v = v / 1e3 if unit in ("ns", "nsecond") else (v * 1e3 if unit in ("ms", "msecond") else v)
            elif d["Metric Name"].startswith("dram__bytes"):
                scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "KB": 1e3, "MB": 1e6, "GB": 1e9}
                v *= scale.get(unit, 1)
            e[3][d["Metric Name"]] = v
    return list(launches.values())


def family(name):
    for k, prefixes in FAMILY.items():
        if name.startswith(prefixes):
            return k
    return None


def summarise(launches, workload):
    starts = [i for i, l in enumerate(launches) if l[0].startswith(STEP_MARKERS)]
    if len(starts) < 2:
        raise SystemExit("fewer than two step markers in the capture")
    # windows between consecutive step markers, leaving out any that contains a prefill
    steps = [(a, b) for a, b in zip(starts[:-1], starts[1:])
             if not any(l[0].startswith("k_prefill") for l in launches[a:b])]
    if not steps:
        raise SystemExit("no complete decode step in the capture")
    agg = collections.OrderedDict()
    fam = {k: [0, 0.0, 0.0] for k in FAMILY}
    total = 0.0
    for a, b in steps:
        for name, grid, block, m in launches[a:b]:
            t = m.get("gpu__time_duration.sum", 0.0)
            total += t
            e = agg.setdefault(f"{name} grid {grid} block {block}", [0, 0.0])
            e[0] += 1
            e[1] += t
            k = family(name)
            if k:
                fam[k][0] += 1
                fam[k][1] += t
                fam[k][2] += m.get("dram__bytes_read.sum", 0.0) + m.get("dram__bytes_write.sum", 0.0)
    ns = len(steps)
    lines = [f"Workload `{workload}`: {ns} complete eager decode steps, "
             f"{sum(b - a for a, b in steps) / ns:.1f} launches and {total / ns:.1f} us of summed device "
             f"time per step (launches serialised under ncu: compare shares, not absolutes).",
             "", "| kernel | launches/step | us/step | share |", "|---|---|---|---|"]
    for k, (c, t) in sorted(agg.items(), key=lambda x: -x[1][1]):
        lines.append(f"| `{k}` | {c / ns:.1f} | {t / ns:.1f} | {100 * t / total:.1f}% |")
    traffic = {}
    has_dram = any("dram__bytes_read.sum" in l[3] for l in launches)
    lines += ["", "| family | launches/step | us/step | share | DRAM bytes/launch |", "|---|---|---|---|---|"]
    for k, (c, t, by) in fam.items():
        per = by / c if c and has_dram else None
        lines.append(f"| {k} | {c / ns:.1f} | {t / ns:.1f} | {100 * t / total:.1f}% | "
                     f"{'%.3e' % per if per is not None else 'n/a'} |")
        if per is not None:
            traffic[k] = {"dram_bytes_per_launch": per, "launches_per_step": c / ns,
                          "source_sha256": source_hash(k)}
    return "\n".join(lines), traffic


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("csv")
    ap.add_argument("--workload", required=True)
    ap.add_argument("--traffic", default=None)
    a = ap.parse_args()
    text, traffic = summarise(load(a.csv), a.workload)
    print(text)
    if a.traffic and traffic:
        d = {}
        if os.path.exists(a.traffic):
            with open(a.traffic) as f:
                d = json.load(f)
        d[a.workload] = traffic
        with open(a.traffic, "w") as f:
            json.dump(d, f, indent=1, sort_keys=True)
            f.write("\n")


if __name__ == "__main__":
    main()
