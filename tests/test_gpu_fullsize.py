"""GPU parity at the workloads' full sizes, in the bench's launch configuration (full batch,
full prompts, the bench's context size and its n, tau and unembedding gains).

The oracle cannot replay a whole batch, so it replays the sampled sequences of each
workload (``oracle_seqs``) one by one, and the GPU rows of those sequences inside the full
batch are compared with it: next-byte and drafter logits within the bf16 tolerance (times
the gain), emitted bytes, t, K and the next c_1 equal. A decision may differ only where the
oracle's margin for that decision is inside the tolerance (a near-tie of the top two logits
of the deciding row, or a drafter probability next to tau); the sequence is then no longer
followed. That the sampled rows equal the
oracle's single-sequence run also shows that sequences of a batch do not interact.
"""
import numpy as np
import pytest

import bench
from oracle import THRESH, IncrementalDecoder, Model
from synth import WORKLOADS, cached_weights, prompts, weight_gains
from synth.configs import load_gains

pytestmark = pytest.mark.gpu

BF16_TOL = 2e-2
STEPS = 16
B1_STEPS = 32
F32_TOL = 1e-4


@pytest.fixture(scope="module")
def lca():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_15454_gb300 import build, lca as mod
    build.build()
    mod.load_library()
    return mod


def _gap(row):
    s = np.sort(row)
    return 0.5 * (s[-1] - s[-2])


def _tau_gap(row, tau):
    mx = row.max()
    lse = mx + np.log(np.exp(row - mx).sum())
    return 0.5 * abs(mx - lse - np.log(tau))


def emitted_margin(rec, tau):
    """Distance, in logit units, of the step's emitted bytes from flipping: the argmax of every
    emitted draft and the tau test of every draft examined (up to the first rejection)."""
    m = np.inf
    mb = np.atleast_2d(rec.mb_logits) if rec.mb_logits is not None else np.zeros((0, 256))
    for i in range(min(rec.a, len(mb))):
        m = min(m, _gap(mb[i]))
    for i in range(min(rec.a + 1, len(mb))):
        m = min(m, _tau_gap(mb[i], tau))
    return m


def next_byte_margin(rec):
    """Distance of the next c_1 (next-byte argmax of the last accepted row) from flipping."""
    return _gap(np.atleast_2d(rec.nb_logits)[rec.a])


_MODELS = {}


def oracle_model(cfg, W):
    """One fp64 oracle model per weight set (the paper-size copy is a few GB)."""
    key = (cfg, id(W))
    if key not in _MODELS:
        _MODELS.clear()
        _MODELS[key] = Model(cfg, W)
    return _MODELS[key]


def column_tol(w, wg, base):
    """Per-column logit tolerance: every logit scales with the gain of its unembedding row, g, and
    g * s for the boundary byte."""
    tol_col = np.full(256, base * wg["gain"])
    tol_col[w.model.boundary_byte] *= wg["space_gain"]
    return tol_col


@pytest.mark.parametrize("name,tau", [("paper_b32", 0.75), ("paper_long_b8", 0.5), ("paper_long_b8", 0.75),
                                      ("paper_long_b8", 0.9), ("mlp_b128", 0.75)])
def test_full_size_sampled_sequences(lca, name, tau):
    w = WORKLOADS[name]
    n = w.n_list[0]
    wg = weight_gains(w, calibrated=w.gain_key in load_gains())
    gain = wg["gain"]
    W = cached_weights(w.model, **wg)
    P = prompts(w, seqs=list(range(w.batch)))
    max_bytes = bench.context_bytes(w, n, bench.DEFAULT_STEPS, bench.DEFAULT_WARMUP,
                                    bench.DEFAULT_PROFILE_STEPS)
    ctx = lca.Context(w.model, W, max_batch=w.batch, max_bytes=max_bytes, max_n=max(n, w.max_n))
    ctx.prefill(P)
    M = oracle_model(w.model, W)
    decs = {}
    for b in w.oracle_seqs:
        d = IncrementalDecoder(M)
        d.prefill(P[b])
        decs[b] = d
    tol_col = column_tol(w, wg, BF16_TOL)
    tol = float(tol_col.max())
    followed = {b: 0 for b in decs}
    for _ in range(STEPS):
        recs = {b: d.step(n, tau, THRESH) for b, d in decs.items()}
        out, cnt = ctx.step(n, tau, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        for b, r in recs.items():
            assert (np.abs(nb[b] - r.nb_logits) <= tol_col).all(), np.abs(nb[b] - r.nb_logits).max()
            if n > 1:
                assert (np.abs(mb[b] - r.mb_logits) <= tol_col).all(), np.abs(mb[b] - r.mb_logits).max()
            if out[b] != r.emitted:
                assert emitted_margin(r, tau) < tol, (b, out[b], r.emitted)
                del decs[b]
                continue
            st = ctx.state(b)
            assert (st["t"], st["K"]) == (r.t, r.K)
            followed[b] += 1
            # the next c_1 (next-byte argmax at the new last position) is a decision of this step
            if st["next_byte"] != int(np.argmax(decs[b].nb_last)):
                assert next_byte_margin(r) < tol, (b, st["next_byte"])
                del decs[b]
        if not decs:
            break
    assert max(followed.values()) >= 2, followed
    # every sequence of the batch advanced by 1..n bytes per step
    for b in range(w.batch):
        assert ctx.state(b)["t"] >= len(P[b]) + min(STEPS, max(followed.values()))
    ctx.close()


@pytest.mark.parametrize("n", [3, 4, 5, 6, 7])
def test_paper_b1_calibrated_steps_with_resync(lca, n):
    """The batch-1 workload exactly as the bench runs it (calibrated gains g and s, the bench's
    context size) for 32 steps: logits within the bf16 tolerance on every step. A decision that
    differs (the emitted bytes, or the next c_1) must have an oracle margin inside the tolerance;
    the GPU is then re-synced to the oracle: a prefill of the oracle's bytes, and the oracle's
    candidates and accepted count forced on the next step (a near-tie of the next c_1 survives a
    prefill). The calibrated regime is checked too: drafts are accepted and segments close."""
    w = WORKLOADS["paper_b1"]
    tau = w.tau_list[0]
    wg = weight_gains(w, calibrated=True)
    W = cached_weights(w.model, **wg)
    p = prompts(w, seqs=[0])[0]
    max_bytes = bench.context_bytes(w, n, bench.DEFAULT_STEPS, bench.DEFAULT_WARMUP, bench.DEFAULT_PROFILE_STEPS)
    ctx = lca.Context(w.model, W, max_batch=1, max_bytes=max_bytes, max_n=max(n, w.max_n))
    ctx.prefill([p])
    dec = IncrementalDecoder(oracle_model(w.model, W))
    dec.prefill(p)
    tol_col = column_tol(w, wg, BF16_TOL)
    tol = float(tol_col.max())
    resync, accepted, K0, force = 0, 0, dec.K, False
    for _ in range(B1_STEPS):
        r = dec.step(n, tau, THRESH)
        if force:
            ctx.force_candidates([bytes([r.c1] + r.drafts)], n)
            ctx.force_accept([r.a])
            force = False
        out, cnt = ctx.step(n, tau, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        assert (np.abs(nb[0] - r.nb_logits) <= tol_col).all(), np.abs(nb[0] - r.nb_logits).max()
        assert (np.abs(mb[0] - r.mb_logits) <= tol_col).all(), np.abs(mb[0] - r.mb_logits).max()
        accepted += r.a
        diverged = out[0] != r.emitted
        if diverged:
            assert emitted_margin(r, tau) < tol, (out[0], r.emitted)
        else:
            st = ctx.state(0)
            assert (st["t"], st["K"]) == (r.t, r.K)
            assert (st["prev_group_start"], st["group_start"]) == dec.group_starts()
            if st["next_byte"] != int(np.argmax(dec.nb_last)):
                assert next_byte_margin(r) < tol
                diverged = True
        if diverged:
            resync += 1
            ctx.prefill([bytes(dec.x)])
            force = True
    assert resync <= B1_STEPS // 8, resync
    assert accepted > 0 and dec.K > K0, (accepted, dec.K, K0)
    ctx.close()


def test_paper_layout_f32_debug_bit_exact(lca):
    """fp32 debug mode at the paper layout (d = 1024, 16 x 64 heads, layers 2/16/2/2, fp32 weights
    and caches, FFMA everywhere) with the calibrated gains: 64 steps whose emitted bytes, accepted
    counts, t, K, open-segment start and group starts equal the oracle's exactly, and whose logits
    agree within 1e-4 times the gain."""
    w = WORKLOADS["paper_b1"]
    model = w.model.replace(dtype="f32")
    n, tau = 4, w.tau_list[0]
    wg = weight_gains(w, calibrated=True)
    W = cached_weights(model, **wg)
    p = prompts(w, seqs=[0])[0]
    ctx = lca.Context(model, W, max_batch=1, max_bytes=len(p) + 64 * n + 16, max_n=n)
    ctx.prefill([p])
    dec = IncrementalDecoder(oracle_model(model, W))
    dec.prefill(p)
    tol_col = column_tol(w, wg, F32_TOL)
    counts, K0 = [], dec.K
    for s in range(64):
        r = dec.step(n, tau, THRESH)
        out, cnt = ctx.step(n, tau, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        assert (np.abs(nb[0] - r.nb_logits) <= tol_col).all(), (s, np.abs(nb[0] - r.nb_logits).max())
        assert (np.abs(mb[0] - r.mb_logits) <= tol_col).all(), (s, np.abs(mb[0] - r.mb_logits).max())
        assert out[0] == r.emitted and int(cnt[0]) == len(r.emitted), (s, out[0], r.emitted, emitted_margin(r, tau))
        st = ctx.state(0)
        assert (st["t"], st["K"], st["open_start"]) == (dec.t, dec.K, dec.open_start())
        assert (st["prev_group_start"], st["group_start"]) == dec.group_starts()
        assert st["next_byte"] == int(np.argmax(dec.nb_last))
        counts.append(r.a)
    assert sum(counts) > 0 and dec.K > K0
    ctx.close()
