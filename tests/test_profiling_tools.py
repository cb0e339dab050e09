"""Host logic of the measurement tools (CPU): the in-graph timeline rebuilt from launch-tracer
records, and the ncu launch-list summary with its per-family DRAM bytes."""
import csv

import numpy as np

from paper_2608_15454_gb300 import ncu_summary, trace_summary

TRACE_DTYPE = [("t0", "<u8"), ("t1", "<u8"), ("tw", "<u8"), ("tag", "<i4"), ("cta", "<i4"), ("sm", "<i4"),
               ("mark", "<i4"), ("mark2", "<i4"), ("mark3", "<i4")]


def _records(rows):
    return np.array([tuple(r) for r in rows], dtype=TRACE_DTYPE)


def test_trace_launches_split_on_tag_change_and_repeated_cta():
    # two GEMV launches back to back (CTA 0 repeats), then an attention launch; given out of order
    rows = [
        (1000, 3000, 1500, 1, 0, 0, 200, 300, 900),
        (1010, 3100, 1500, 1, 1, 1, 210, 310, 910),
        (2000, 5000, 3200, 1, 0, 2, 300, 400, 1000),
        (2020, 5200, 3200, 1, 1, 3, 300, 420, 1100),
        (4000, 9000, 5300, 5, 0, 4, 0, 0, 0),
    ]
    rec = _records([rows[i] for i in (4, 2, 0, 3, 1)])
    L = trace_summary.launches(rec)
    assert [trace_summary.TAGS[x["tag"]] for x in L] == ["gemv", "gemv", "attn"]
    assert [len(x["recs"]) for x in L] == [2, 2, 1]
    s = trace_summary.summarise(rec)
    assert s[0]["wait_us"] == 0.5 and s[0]["end_us"] == 2.1       # from the first entry (t0 = 1000 ns)
    assert s[1]["incr_us"] == (5200 - 3200) / 1e3                 # after its own first wait
    # phases of the first GEMV: wait -> staged -> weights -> dots -> exit (medians over its 2 CTAs)
    ph = s[0]["phases_us"]
    assert list(ph) == ["staged", "weights", "dots", "exit"]
    np.testing.assert_allclose(ph["weights"], 0.1)
    np.testing.assert_allclose(sum(ph.values()), np.median([3000 - 1500, 3100 - 1500]) / 1e3, atol=1e-9)
    assert "phases_us" not in s[2]                                # no marks recorded


def _write_launch_csv(path, launches):
    hdr = ["ID", "Kernel Name", "Grid Size", "Block Size", "Metric Name", "Metric Unit", "Metric Value"]
    with open(path, "w", newline="") as f:
        w = csv.writer(f)
        w.writerow(hdr)
        for i, (name, grid, ns, dram_mb) in enumerate(launches):
            w.writerow([i, f"void lca::<unnamed>::{name}(Dev)", grid, "(128, 1, 1)", "gpu__time_duration.sum",
                        "nsecond", f"{ns:,}"])
            w.writerow([i, f"void lca::<unnamed>::{name}(Dev)", grid, "(128, 1, 1)", "dram__bytes_read.sum",
                        "Mbyte", dram_mb])


def test_ncu_summary_steps_shares_and_family_bytes(tmp_path):
    step = [("k_mb_plan", "(1, 1, 1)", 2000, 0.0), ("k_gemv_bulk<1, 4, 1>", "(192, 1, 1)", 6000, 6.0),
            ("k_attn_w<4>", "(1, 1, 256)", 10000, 1.5), ("k_gemv_bulk<1, 4, 0>", "(64, 4, 1)", 4000, 2.0),
            ("k_commit", "(1, 1, 1)", 3000, 0.0)]
    p = tmp_path / "launches.csv"
    _write_launch_csv(p, step * 3 + step[:1])          # three complete steps, then the next step's start
    launches = ncu_summary.load(str(p))
    assert len(launches) == 16 and launches[1][0] == "k_gemv_bulk<1, 4, 1>"
    assert launches[1][3]["gpu__time_duration.sum"] == 6.0          # ns -> us
    assert launches[1][3]["dram__bytes_read.sum"] == 6.0e6          # Mbyte -> bytes
    text, traffic = ncu_summary.summarise(launches, "w")
    assert "3 complete eager decode steps, 5.0 launches and 25.0 us" in text
    assert "| `k_attn_w<4> grid (1, 1, 256) block (128, 1, 1)` | 1.0 | 10.0 | 40.0% |" in text
    assert traffic["linear"]["launches_per_step"] == 2.0
    np.testing.assert_allclose(traffic["linear"]["dram_bytes_per_launch"], 4.0e6)
    np.testing.assert_allclose(traffic["attention"]["dram_bytes_per_launch"], 1.5e6)
    assert len(traffic["linear"]["source_sha256"]) == 64
