"""The bench's algorithmic-byte accounting (CPU), against the sizes the model's shape fixes:
one pre-norm Llama block of width d with a 4d SwiGLU MLP holds 16 d^2 weights (Q, K, V, O:
4 d^2; W1, W3, W2: 12 d^2), 33.55 MB in bf16 at d = 1024, and the paper-size model runs
2 encoder + 2 next-byte + 2 multi-byte blocks every step and 16 LM blocks when a patch closes."""
import numpy as np

import bench
from synth import WORKLOADS

MB = 1e6


def _stats(steps, lm_steps, lm_rows):
    return {"steps": steps, "lm_steps": lm_steps, "lm_rows": lm_rows}


def _state(t, K, pgs):
    return {"t": t, "K": K, "prev_group_start": pgs}


def test_weight_bytes_per_step_of_the_paper_model():
    m = WORKLOADS["paper_b1"].model
    blk = 16 * 1024 * 1024 * 2
    assert abs(blk / MB - 33.55) < 0.01
    unembed = 256 * 1024 * 2
    s0 = [_state(1000, 130, 990)]
    # no LM step: 6 blocks and the two heads' unembedding
    w, _ = bench.algorithmic_bytes(m, 3, 10, _stats(0, 0, 0), _stats(10, 0, 0), s0, s0)
    assert w == 6 * blk + 2 * unembed
    assert abs(w / MB - 202.4) < 0.1
    # every step runs the LM module: 22 blocks, about 738 MB
    w, _ = bench.algorithmic_bytes(m, 3, 10, _stats(0, 0, 0), _stats(10, 10, 10), s0, s0)
    assert w == 22 * blk + 2 * unembed
    assert abs(w / MB - 739.2) < 0.1
    # n = 1: no drafter, one head
    w, _ = bench.algorithmic_bytes(m, 1, 10, _stats(0, 0, 0), _stats(10, 0, 0), s0, s0)
    assert w == 4 * blk + unembed


def test_kv_bytes_per_step_of_the_paper_model():
    """Byte caches: K and V of every encoder and next-byte layer read once at the mid-interval
    length (16 KB per position over 4 layers: 1024 dims x 2 B x 2 x 4), plus the n appended rows;
    the window cache of the two multi-byte layers; the LM cache (64 KB per latent over 16 layers)
    for each new latent row."""
    m = WORKLOADS["paper_b1"].model
    n = 3
    a, b = _state(1000, 130, 990), _state(1030, 134, 1020)
    _, kv = bench.algorithmic_bytes(m, n, 10, _stats(0, 0, 0), _stats(10, 2, 4), [a], [b])
    per_pos = 1024 * 2 * 2               # K and V of one layer at one position
    t_mid, win, k_mid = 1015.0, 10.0, 132.0
    byte_read = 4 * per_pos * (t_mid + n)
    byte_append = 4 * per_pos * n
    window = 2 * per_pos * (win + n)
    lm = 0.4 * 16 * per_pos * (k_mid + 2)   # 4 LM rows over 10 steps
    assert np.isclose(kv, byte_read + byte_append + window + lm)
    assert per_pos * 4 == 16384 and per_pos * 16 == 65536


def test_roofline_of_the_dominant_family():
    """The family's in-graph time is its share of the eager kernel time times the graph step time,
    so the families add up to the step; achieved = algorithmic bytes per launch over that time."""
    prof = {"linear": {"launches": 88, "ms": 0.264, "bytes": 88 * 8.39e6},
            "attention": {"launches": 22, "ms": 0.110, "bytes": 0.0},
            "head": {"launches": 2, "ms": 0.026, "bytes": 0.0}}
    steps, ms_per_step = 2, 0.1  # graph: 0.1 ms/step against 0.2 ms/step of eager kernel time
    r = bench.roofline(prof, 6670.9, "measured", "nowhere", 1.0e6, steps, ms_per_step)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == 6670.9
    share = 0.264 / 0.4
    assert np.isclose(r["share_of_step"], share)
    per_launch_s = share * ms_per_step * 1e-3 * steps / 88
    assert np.isclose(r["achieved"], 8.39e6 / per_launch_s / 1e9)
    assert np.isclose(r["frac"], r["achieved"] / 6670.9)
    assert r["traffic"] is None
    # the implied kernel time per step never exceeds the step
    assert r["in_graph_us_per_launch"] * r["launches_per_step"] <= ms_per_step * 1e3 + 1e-9
    # attention dominant: its bytes per launch are the step KV bytes times the steps, per launch
    prof["attention"]["ms"] = 1.0
    r = bench.roofline(prof, 6670.9, "measured", "nowhere", 1.0e6, steps, ms_per_step)
    assert np.isclose(r["algorithmic_bytes_per_launch"], 2 * 1.0e6 / 22)


def test_blocks_and_context_size():
    assert bench.blocks_of(20) == [20]
    assert bench.blocks_of(130) == [64, 64, 2]
    assert sum(bench.blocks_of(512)) == 512
    w = WORKLOADS["paper_b1"]
    # a block, the warm-up or the profiled steps after one prefill, each at most n bytes a step
    assert bench.context_bytes(w, 7, 512, 5, 20) == 1024 + (64 + 2) * 7 + 8
    assert bench.context_bytes(w, 3, 20, 5, 20) == 1024 + (20 + 2) * 3 + 8


def test_sweep_covers_the_rest_of_the_metric():
    class A:
        sweep, batch, prompt_bytes = "auto", None, None
    cases = bench.sweep_cases(WORKLOADS["paper_b1"], 3, A)
    assert cases == [("paper_b1", 4), ("paper_b1", 5), ("paper_b1", 6), ("paper_b1", 7), ("paper_b32", 4)]
    A.sweep = "none"
    assert bench.sweep_cases(WORKLOADS["paper_b1"], 3, A) == []


def test_prefill_flops_of_the_paper_model():
    """Linear FLOPs: 2 x 16 d^2 per row per block (32 d^2 = 33.6 MFLOP at d = 1024); the byte
    modules see every byte, the LM module every latent plus BOS; causal attention 2 d T (T + 1)
    per byte layer."""
    m = WORKLOADS["paper_b1"].model
    p = b"ab cd"  # 5 bytes, one boundary: 2 latent rows
    d = 1024
    lin = 2 * 16 * d * d * (5 * 4 + 2 * 16)
    att = 2 * d * 5 * 6 * 4 + 2 * d * 2 * 3 * 16
    assert bench.prefill_flops(m, [p]) == lin + att + 2 * 256 * d


def test_reference_arm_times_the_oracle_steps():
    """`bench.py --impl reference` runs the oracle alone (no GPU): K timed decode steps after W
    untimed ones, one JSON line with the arm's metric, e2e without copies and its cpu_baseline."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny_b1",
                        "--steps", "4", "--warmup", "3"], cwd=root, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "bytes/s" and line["higher_is_better"]
    assert line["steps"] == 4 and line["warmup"] == 3 and line["value"] > 0 and line["ms_per_step"] > 0
    assert line["e2e"] == {"value": line["value"], "unit": "bytes/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["cores"] >= 1
    assert "4 timed decode steps" in cb["sample"] and "3 untimed steps" in cb["sample"]
    assert line["config"]["workload"] == "tiny_b1"


def test_reference_arm_runs_on_rank_zero_only():
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny_b1",
                        "--gpus", "2", "--steps", "2", "--warmup", "3"], cwd=root, env=env,
                       capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == ""
