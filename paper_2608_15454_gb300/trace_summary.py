"""In-graph timeline of the decode step from the library's launch tracer.

`lca_debug_trace` runs decode steps as the step graph (programmatic dependent launch included)
while thread 0 of every CTA records its entry time, the time its grid-dependency wait returned,
up to three mid-kernel marks and its exit time (device globaltimer). This script rebuilds the
launches from those records and prints, per launch, when its first CTA passed the dependency wait
(the predecessor had completed), when its last CTA exited, and the median over CTAs of the phases
between the marks:

* k_gemv_bulk: wait -> rows staged (bf16 halves) -> weights in shared memory -> dot products
  summed -> exit;
* k_attn_w: wait -> staged keys landed -> key loop done -> split partials combined -> exit.

    python -m paper_2608_15454_gb300.trace_summary --workload paper_b1 [--warm 200] [--steps 3]

Needs a GPU and a bf16 workload. Launches are rebuilt from the records: a launch's CTAs all start
before any CTA of the next launch (each kernel triggers its dependents at entry), so a new launch
begins where the kernel tag changes or a CTA index repeats.
"""
from __future__ import annotations

import argparse
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

TAGS = {1: "gemv", 2: "gemv_f32", 3: "gemm", 4: "rowstats", 5: "attn", 6: "head", 7: "mb_plan",
        8: "mb_fill", 9: "mlp_plan", 10: "verify_plan", 11: "segment", 12: "lm_scatter",
        13: "nb_input", 14: "commit", 15: "loop_ctl", 16: "other", 17: "umma", 18: "split", 19: "sgemm", 20: "stack"}
PHASES = {"gemv": ("staged", "weights", "dots", "exit"), "attn": ("keys landed", "key loop", "combined", "exit")}


def launches(rec):
    """Group trace records (any order) into launches in start order."""
    r = rec[np.argsort(rec["t0"], kind="stable")]
    out, cur = [], None
    for x in r:
        tag, cta = int(x["tag"]), int(x["cta"])
        if cur is None or cur["tag"] != tag or cta in cur["ctas"]:
            cur = {"tag": tag, "ctas": set(), "recs": []}
            out.append(cur)
        cur["ctas"].add(cta)
        cur["recs"].append(x)
    for L in out:
        L["recs"] = np.array(L["recs"], dtype=rec.dtype)
    return out


def summarise(rec):
    """One dict per launch: tag, CTAs, first wait, end (us from the first launch's start),
    increment over the previous launch's end, and median phase times (us) where marked."""
    Ls = launches(rec)
    if not Ls:
        return []
    base = int(Ls[0]["recs"]["t0"].min())
    prev_end = base
    rows = []
    for L in Ls:
        R = L["recs"]
        t0 = R["t0"].astype(np.int64)
        tw = R["tw"].astype(np.int64)
        t1 = R["t1"].astype(np.int64)
        marks = [R[f].astype(np.int64) for f in ("mark", "mark2", "mark3")]
        tag = TAGS.get(L["tag"], str(L["tag"]))
        first_wait, end = int(tw.min()), int(t1.max())
        row = {"tag": tag, "ctas": len(R), "wait_us": (first_wait - base) / 1e3, "end_us": (end - base) / 1e3,
               "incr_us": (end - max(prev_end, first_wait)) / 1e3}
        if tag in PHASES and all(m.max() > 0 for m in marks):
            edges = [tw - t0] + marks + [t1 - t0]
            row["phases_us"] = {name: float(np.median(edges[i + 1] - edges[i])) / 1e3
                                for i, name in enumerate(PHASES[tag])}
        rows.append(row)
        prev_end = max(prev_end, end)
    return rows


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="paper_b1")
    ap.add_argument("--n", type=int, default=None)
    ap.add_argument("--warm", type=int, default=200, help="untimed decode steps before the trace")
    ap.add_argument("--steps", type=int, default=3)
    a = ap.parse_args()
    import torch  # noqa: F401  (device memory of the context)
    from paper_2608_15454_gb300 import build, lca
    from synth import WORKLOADS, cached_weights, prompts, weight_gains
    build.build()
    w = WORKLOADS[a.workload]
    n = a.n or w.n_list[0]
    tau = w.tau_list[0]
    wg = weight_gains(w, True)
    W = cached_weights(w.model, **wg)
    P = prompts(w, seqs=list(range(w.batch)))
    ctx = lca.Context(w.model, W, max_batch=w.batch, max_bytes=w.prompt_len + (a.warm + a.steps + 4) * n + 64,
                      max_n=max(n, w.max_n), device="cuda:0")
    ctx.prefill(P)
    for _ in range(a.warm):
        ctx.step_async(n, tau, lca.LCA_THRESH)
    rec = ctx.trace(n, tau, lca.LCA_THRESH, a.steps)
    ctx.close()
    rows = summarise(rec)
    print(f"{a.workload} n={n}: {len(rows)} launches in {a.steps} traced steps after {a.warm} steps")
    print("| launch | CTAs | first wait (us) | end (us) | increment (us) | median phases (us) |")
    print("|---|---|---|---|---|---|")
    for r in rows:
        ph = ", ".join(f"{k} {v:.2f}" for k, v in r.get("phases_us", {}).items())
        print(f"| {r['tag']} | {r['ctas']} | {r['wait_us']:.2f} | {r['end_us']:.2f} | {r['incr_us']:.2f} | {ph} |")


if __name__ == "__main__":
    main()
