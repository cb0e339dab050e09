"""Choose the two unembedding gains of each synthetic model on the oracle, and write them to
``synth/gains.json``.

TEST INFRASTRUCTURE ONLY: it runs the CPU oracle and nothing else.

Random-init weights give near-uniform byte distributions, so at tau = 0.75 no draft passes, and
the greedy text they generate holds no spaces, so no segment ever closes and the LM module never
runs: neither is the regime the paper measures. Two deterministic changes to the unembedding
W_u bring the decode loop to the paper's regime without changing the method:

  * g multiplies all of W_u. It changes no argmax (up to bf16 rounding) and only sharpens the
    softmax, which sets the acceptance rate. The paper's trained models accept about half of
    the drafted bytes (Section 5, byte acceptance rates; Section 6.2, mean 3.05 of 6 drafts
    accepted per step); the target is a mean a / (n - 1) of 0.5.
  * s multiplies the boundary byte's row of W_u (before g). It raises how often a space wins
    the argmax; the target is the space rate of the workload's own prompts (one segment per
    word), so that segments close, and the LM module runs, about as often as on real text.

Each gain is found by bisection on its logarithm over the first ``steps`` decode steps of
sequence 0 of the named workload (threshold acceptance), alternating g and s twice.

    python oracle/calibrate_gain.py [--keys paper paper_mlp tiny] [--steps 64]
"""
from __future__ import annotations

import argparse
import json
import math
import os
import sys
import time

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

from oracle.decode import THRESH, IncrementalDecoder  # noqa: E402
from oracle.model import Model  # noqa: E402
from synth import WORKLOADS, make_weights, prompt  # noqa: E402
from synth.configs import _GAINS_PATH  # noqa: E402

# key -> (workload whose model and prompt are used, n, tau)
TARGETS = {
    "tiny": ("tiny_b1", 3, 0.75),
    "paper": ("paper_b1", 5, 0.75),
    "paper_mlp": ("mlp_b128", 7, 0.75),
}


def run(workload, n, tau, gain, space_gain, steps):
    """(acceptance, space rate of the emitted bytes) over the first `steps` decode steps."""
    w = WORKLOADS[workload]
    M = Model(w.model, make_weights(w.model, gain=gain, space_gain=space_gain))
    dec = IncrementalDecoder(M)
    dec.prefill(prompt(w, 0))
    acc = emitted = spaces = 0
    for _ in range(steps):
        r = dec.step(n, tau, THRESH)
        acc += r.a
        emitted += len(r.emitted)
        spaces += r.emitted.count(bytes([w.model.boundary_byte]))
    return acc / (steps * (n - 1)), spaces / max(1, emitted)


def _dist(v, target):
    return abs(math.log(max(v, 1e-6) / target))


def bisect(evaluate, lo, hi, target, iters, log):
    """Bisection on log x in [lo, hi] for evaluate(x) ~ target (evaluate increasing in x);
    returns the x whose value is closest to the target in ratio, and that value. The space rate
    of greedy text jumps between attractors (no spaces at all, or a word-like rhythm), so the
    distance is |log(value / target)|: a rate of 0 is never the closest."""
    best = None
    a, b = math.log(lo), math.log(hi)
    for _ in range(iters):
        mid = 0.5 * (a + b)
        x = round(math.exp(mid), 4)
        v = evaluate(x)
        log(f"  x={x} -> {v:.3f}")
        if best is None or _dist(v, target) < _dist(best[1], target):
            best = (x, v)
        if v < target:
            a = mid
        else:
            b = mid
    return best


def calibrate(key, steps, iters, log):
    workload, n, tau = TARGETS[key]
    w = WORKLOADS[workload]
    p = prompt(w, 0)
    space_target = p.count(bytes([w.model.boundary_byte])) / len(p)
    g, s = 8.0, 1.0
    g_lo, g_hi, s_lo, s_hi = 1.0, 4096.0, 1.0, 64.0
    for rnd in range(2):
        t0 = time.time()
        log(f"{key}: round {rnd}, gain for acceptance 0.5 (space gain {s})")
        g, acc = bisect(lambda x: run(workload, n, tau, x, s, steps)[0], g_lo, g_hi, 0.5, iters, log)
        log(f"{key}: space gain for space rate {space_target:.3f} (gain {g})")
        s, rate = bisect(lambda x: run(workload, n, tau, g, x, steps)[1], s_lo, s_hi, space_target, iters, log)
        g_lo, g_hi = g / 4, g * 4
        s_lo, s_hi = max(1.0, s / 4), s * 4
        log(f"{key}: round {rnd}: gain {g}, space gain {s} ({time.time() - t0:.0f} s)")
    acc, rate = run(workload, n, tau, g, s, steps)
    return {"gain": g, "space_gain": s, "acceptance": round(acc, 4), "space_rate": round(rate, 4),
            "space_rate_target": round(space_target, 4), "workload": workload, "n": n, "tau": tau,
            "steps": steps, "target": 0.5}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--keys", nargs="*", default=list(TARGETS))
    ap.add_argument("--steps", type=int, default=64)
    ap.add_argument("--iters", type=int, default=7)
    a = ap.parse_args()
    gains = {}
    if os.path.exists(_GAINS_PATH):
        with open(_GAINS_PATH) as f:
            gains = json.load(f)
    for key in a.keys:
        gains[key] = calibrate(key, a.steps, a.iters, lambda s: print(s, flush=True))
        with open(_GAINS_PATH, "w") as f:
            json.dump(gains, f, indent=1, sort_keys=True)
            f.write("\n")
    print(json.dumps(gains))


if __name__ == "__main__":
    main()
