"""Choose the unembedding gain g of each synthetic model on the oracle, and write it to
``synth/gains.json``.

TEST INFRASTRUCTURE ONLY: it runs the CPU oracle and nothing else.

Random-init weights give near-uniform byte distributions, so at tau = 0.75 no draft
passes and the decode step degenerates to one byte per step. The paper's trained models
accept about half of the drafted bytes (Section 5, byte acceptance rates; Section 6.2,
mean 3.05 of 6 drafts accepted per step). Scaling the unembedding, W_u <- g * W_u,
changes no argmax (up to bf16 rounding) and only sharpens the softmax, so one scalar per
model sets the acceptance rate. g is found by bisection on log g: the first ``steps``
decode steps of sequence 0 of the named workload, threshold acceptance, target mean
a / (n - 1) = 0.5.

    python oracle/calibrate_gain.py [--keys tiny paper paper_mlp] [--steps 64]
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


def acceptance(workload, n, tau, gain, steps):
    w = WORKLOADS[workload]
    M = Model(w.model, make_weights(w.model, gain=gain))
    dec = IncrementalDecoder(M)
    dec.prefill(prompt(w, 0))
    acc = 0
    for _ in range(steps):
        acc += dec.step(n, tau, THRESH).a
    return acc / (steps * (n - 1))


def calibrate(key, steps, iters, log):
    workload, n, tau = TARGETS[key]
    lo, hi = 0.0, math.log(4096.0)          # bracket on log g
    best = None
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        g = round(math.exp(mid), 3)
        t0 = time.time()
        r = acceptance(workload, n, tau, g, steps)
        log(f"{key}: g={g} acceptance={r:.3f} ({time.time() - t0:.0f} s)")
        if best is None or abs(r - 0.5) < abs(best[1] - 0.5):
            best = (g, r)
        if r < 0.5:
            lo = mid
        else:
            hi = mid
    g, r = best
    return {"gain": g, "acceptance": round(r, 4), "workload": workload, "n": n, "tau": tau,
            "steps": steps, "target": 0.5}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--keys", nargs="*", default=list(TARGETS))
    ap.add_argument("--steps", type=int, default=64)
    ap.add_argument("--iters", type=int, default=10)
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
