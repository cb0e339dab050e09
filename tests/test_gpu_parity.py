"""GPU parity: the CUDA decode step through the C ABI against the CPU oracle.

fp32 storage (the tiny model): committed bytes, accepted counts, t, K and group starts
bit-exact; next-byte and drafter logits within 1e-4 (times the unembedding gain).
bf16 storage (the paper-size model): logits within 2e-2; decisions compared with a
teacher-forced re-sync: at a divergent decision the oracle's margin must be below the
tolerance, then both continue from the oracle's bytes.
"""
import numpy as np
import pytest

from oracle import SPEC, THRESH, IncrementalDecoder, Model
from synth import TINY, WORKLOADS, cached_weights, make_weights, prompt, words_text, zipf_text

pytestmark = pytest.mark.gpu

F32_TOL = 1e-4
BF16_TOL = 2e-2


@pytest.fixture(scope="module")
def lca():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_15454_gb300 import build, lca as mod
    build.build()
    mod.load_library()
    return mod


def new_ctx(lca, model, weights, batch, max_bytes, max_n):
    return lca.Context(model, weights, max_batch=batch, max_bytes=max_bytes, max_n=max_n)


def check_step(ctx, dec_list, recs, n, tol, out, cnt, exact=True):
    nb, mb = ctx.logits(n)
    for b, (dec, r) in enumerate(zip(dec_list, recs)):
        np.testing.assert_allclose(nb[b], r.nb_logits, atol=tol, rtol=0)
        if n > 1:
            np.testing.assert_allclose(mb[b], r.mb_logits, atol=tol, rtol=0)
        if exact:
            assert out[b] == r.emitted, (b, out[b], r.emitted)
            assert cnt[b] == len(r.emitted)
            st = ctx.state(b)
            assert (st["t"], st["K"]) == (dec.t, dec.K)
            assert st["open_start"] == dec.open_start()
            assert (st["prev_group_start"], st["group_start"]) == dec.group_starts()


# ----------------------------------------------------------------------------- tiny fp32
def test_tiny_generate_matches_oracle_bytes(lca):
    w = WORKLOADS["tiny_b1"]
    W = cached_weights(w.model)
    p = prompt(w, 0)
    ctx = new_ctx(lca, w.model, W, 1, w.max_bytes, w.max_n)
    ctx.prefill([p])
    out, hist = ctx.generate(3, 0.75, lca.LCA_THRESH, w.gen)
    from oracle import generate_incremental
    want, recs = generate_incremental(Model(w.model, W), p, 3, 0.75, THRESH, w.gen)
    assert out[0] == want
    assert hist.sum() == len(recs)
    assert ctx.state(0)["t"] == len(p) + w.gen


@pytest.mark.parametrize("gain,mode,tau", [(1.0, THRESH, 0.75), (40.0, THRESH, 0.5), (40.0, SPEC, 0.75)])
def test_tiny_steps_logits_and_state(lca, gain, mode, tau):
    w = WORKLOADS["tiny_b1"]
    W = make_weights(w.model, gain=gain)
    p = prompt(w, 0)
    n = 4
    ctx = new_ctx(lca, w.model, W, 1, len(p) + 200, 8)
    ctx.prefill([p])
    dec = IncrementalDecoder(Model(w.model, W))
    dec.prefill(p)
    acc = 0
    for _ in range(30):
        out, cnt = ctx.step(n, tau, mode)
        r = dec.step(n, tau, mode)
        acc += r.a
        check_step(ctx, [dec], [r], n, F32_TOL * gain, out, cnt)
    if gain > 1 and mode == THRESH:
        assert acc > 0


def test_tiny_forced_boundaries_and_rollback(lca):
    """Candidates holding spaces at every place, with forced accepted counts: the LM module
    runs on speculative segments and the rejected ones are rolled back."""
    w = WORKLOADS["tiny_b1"]
    W = cached_weights(w.model)
    p = prompt(w, 0)
    n = 4
    pats = [b"ab c", b" abc", b"a  b", b"    ", b"abcd", b"x y ", b"  xy", b"q   "]
    forced = [0, 3, 1, 2, 3, 0, 2, 1, 3, 3, 0]
    ctx = new_ctx(lca, w.model, W, 1, len(p) + 200, n)
    ctx.prefill([p])
    dec = IncrementalDecoder(Model(w.model, W))
    dec.prefill(p)
    for s in range(40):
        cand, a = pats[s % len(pats)], forced[s % len(forced)]
        ctx.force_candidates([cand], n)
        ctx.force_accept([a])
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        r = dec.step(n, 0.75, THRESH, forced=a, forced_cand=cand)
        check_step(ctx, [dec], [r], n, F32_TOL, out, cnt)
        # a free step after each forced one exercises the rebuilt multi-byte window
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        r = dec.step(n, 0.75, THRESH)
        check_step(ctx, [dec], [r], n, F32_TOL, out, cnt)


def test_tiny_ragged_batch_equals_sequences_alone(lca):
    model = TINY
    W = cached_weights(model)
    prompts = [words_text(0, 200), words_text(1, 57) + b" ", words_text(2, 131), b"a"]
    n = 3
    ctx = new_ctx(lca, model, W, len(prompts), 400, n)
    ctx.prefill(prompts)
    decs = []
    for p in prompts:
        d = IncrementalDecoder(Model(model, W))
        d.prefill(p)
        decs.append(d)
    for s in range(20):
        a = [s % 3, (s + 1) % 3, 2, 0]
        cands = [bytes([97 + (s + b) % 26, 32 if (s + b) % 3 == 0 else 98, 99]) for b in range(len(prompts))]
        if s % 2 == 0:
            ctx.force_candidates(cands, n)
            ctx.force_accept(a)
            recs = [d.step(n, 0.75, THRESH, forced=a[b], forced_cand=cands[b]) for b, d in enumerate(decs)]
        else:
            recs = [d.step(n, 0.75, THRESH) for d in decs]
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        check_step(ctx, decs, recs, n, F32_TOL, out, cnt)


def test_tiny_mlp_head(lca):
    model = TINY.replace(mb_kind="mlp", n_mb=3, n_mlp_heads=4)
    W = make_weights(model, gain=40.0)
    p = words_text(3, 180)
    n = 5
    ctx = new_ctx(lca, model, W, 1, 400, n)
    ctx.prefill([p])
    dec = IncrementalDecoder(Model(model, W))
    dec.prefill(p)
    for _ in range(20):
        out, cnt = ctx.step(n, 0.5, lca.LCA_THRESH)
        r = dec.step(n, 0.5, THRESH)
        check_step(ctx, [dec], [r], n, F32_TOL * 40, out, cnt)


def test_tiny_n1_and_generate_budget(lca):
    w = WORKLOADS["tiny_b1"]
    W = make_weights(w.model, gain=40.0)
    p = prompt(w, 0)
    ctx = new_ctx(lca, w.model, W, 1, len(p) + 100, 5)
    ctx.prefill([p])
    out1, _ = ctx.generate(1, 0.75, lca.LCA_THRESH, 20)
    ctx.prefill([p])
    out5, hist = ctx.generate(5, 0.0, lca.LCA_THRESH, 23)
    from oracle import generate_incremental
    M = Model(w.model, W)
    assert out1[0] == generate_incremental(M, p, 1, 0.75, THRESH, 20)[0]
    want, recs = generate_incremental(M, p, 5, 0.0, THRESH, 23)
    assert out5[0] == want and len(out5[0]) == 23
    assert hist[4] == len(recs)   # tau = 0 accepts every draft


# ----------------------------------------------------------------------------- paper bf16
def _margin(logits):
    s = np.sort(logits)
    return s[-1] - s[-2]


@pytest.mark.parametrize("n", [3, 7])
def test_paper_bf16_steps_with_resync(lca, n):
    w = WORKLOADS["paper_b1"]
    W = cached_weights(w.model)
    p = prompt(w, 0)
    ctx = new_ctx(lca, w.model, W, 1, w.max_bytes, 7)
    ctx.prefill([p])
    dec = IncrementalDecoder(Model(w.model, W))
    dec.prefill(p)
    resync = 0
    for s in range(6):
        cand = None
        if s % 2 == 1:   # drive a boundary through the step
            cand = bytes([32 if i == 1 else 101 + i for i in range(n)])
            ctx.force_candidates([cand], n)
            ctx.force_accept([min(2, n - 1)])
            r = dec.step(n, 0.75, THRESH, forced=min(2, n - 1), forced_cand=cand)
        else:
            r = dec.step(n, 0.75, THRESH)
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        np.testing.assert_allclose(nb[0], r.nb_logits, atol=BF16_TOL, rtol=0)
        np.testing.assert_allclose(mb[0], r.mb_logits, atol=BF16_TOL, rtol=0)
        if out[0] != r.emitted:
            rows = np.concatenate([r.mb_logits, r.nb_logits])
            assert min(_margin(x) for x in rows) < 2 * BF16_TOL
            resync += 1
            ctx.prefill([bytes(dec.x)])
        st = ctx.state(0)
        assert (st["t"], st["K"]) == (dec.t, dec.K)
    assert resync <= 1


# ----------------------------------------------------------------------------- small bf16
SMALL_BF16 = TINY.replace(d_model=256, n_heads=4, head_dim=64, d_ff=1024, n_enc=1, n_lm=2,
                          n_nb=1, n_mb=2, dtype="bf16")


@pytest.mark.parametrize("mb_kind", ["lca", "mlp"])
def test_small_bf16_batch_forced_and_free_steps(lca, mb_kind):
    """bf16 storage at d = 256 (bulk-copy weight pipeline, split-K and grouped paths): logits
    within the bf16 tolerance, and bytes/state equal whenever the oracle's decisions have margin."""
    model = SMALL_BF16 if mb_kind == "lca" else SMALL_BF16.replace(mb_kind="mlp", n_mb=3, n_mlp_heads=5)
    W = make_weights(model, gain=8.0, seed=5)
    prompts = [zipf_text(0, 300), zipf_text(1, 77) + b" ", zipf_text(2, 150)]
    n = 4
    ctx = new_ctx(lca, model, W, len(prompts), 600, 6)
    ctx.prefill(prompts)
    decs = []
    for p in prompts:
        d = IncrementalDecoder(Model(model, W))
        d.prefill(p)
        decs.append(d)
    for s in range(12):
        cands = [bytes([97 + (s + b) % 26, 32 if (s + b) % 2 == 0 else 98, 99, 32]) for b in range(3)]
        a = [s % 4, (s + 2) % 4, 3]
        ctx.force_candidates(cands, n)
        ctx.force_accept(a)
        recs = [d.step(n, 0.75, THRESH, forced=a[b], forced_cand=cands[b]) for b, d in enumerate(decs)]
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        for b, r in enumerate(recs):
            np.testing.assert_allclose(nb[b], r.nb_logits, atol=BF16_TOL * 8, rtol=0)
            np.testing.assert_allclose(mb[b], r.mb_logits, atol=BF16_TOL * 8, rtol=0)
            assert out[b] == r.emitted
            st = ctx.state(b)
            assert (st["t"], st["K"]) == (decs[b].t, decs[b].K)


def test_small_bf16_long_context_batch_one(lca):
    """Batch 1 over a cache longer than the decode attention stages in shared memory (about 8,500
    bytes in 16 key splits: 256 staged keys per CTA, the rest read from the cache) and a latent
    cache of about a thousand latents; forced spaces run the LM module on some steps. Logits within
    the bf16 tolerance, bytes and state equal."""
    W = make_weights(SMALL_BF16, gain=8.0, seed=6)
    p = zipf_text(3, 8500)
    n = 3
    ctx = new_ctx(lca, SMALL_BF16, W, 1, len(p) + 64, n)
    ctx.prefill([p])
    dec = IncrementalDecoder(Model(SMALL_BF16, W))
    dec.prefill(p)
    for s in range(6):
        cand = bytes([32 if s % 2 == 0 else 100, 101 + s, 32 if s % 3 == 0 else 102])
        a = s % n
        ctx.force_candidates([cand], n)
        ctx.force_accept([a])
        r = dec.step(n, 0.75, THRESH, forced=a, forced_cand=cand)
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        np.testing.assert_allclose(nb[0], r.nb_logits, atol=BF16_TOL * 8, rtol=0)
        np.testing.assert_allclose(mb[0], r.mb_logits, atol=BF16_TOL * 8, rtol=0)
        assert out[0] == r.emitted
        st = ctx.state(0)
        assert (st["t"], st["K"]) == (dec.t, dec.K)


@pytest.mark.parametrize("mb_kind", ["lca", "mlp"])
def test_persistent_stack_kernel_matches_oracle(lca, mb_kind, monkeypatch):
    """The persistent block-stack kernel (LCA_PERSIST=1: every block of a module in one launch, grid
    barriers between the phases, split-on-write inputs staged by bulk copies) against the oracle at
    d = 256 with forced boundaries: logits within the bf16 tolerance, bytes and state equal."""
    monkeypatch.setenv("LCA_PERSIST", "1")
    model = SMALL_BF16 if mb_kind == "lca" else SMALL_BF16.replace(mb_kind="mlp", n_mb=3, n_mlp_heads=5)
    W = make_weights(model, gain=8.0, seed=5)
    prompts = [zipf_text(0, 300)]
    n = 4
    ctx = new_ctx(lca, model, W, 1, 600, 6)
    ctx.prefill(prompts)
    dec = IncrementalDecoder(Model(model, W))
    dec.prefill(prompts[0])
    for s in range(10):
        cand = bytes([97 + s % 26, 32 if s % 2 == 0 else 98, 99, 32])
        ctx.force_candidates([cand], n)
        ctx.force_accept([s % 4])
        r = dec.step(n, 0.75, THRESH, forced=s % 4, forced_cand=cand)
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        np.testing.assert_allclose(nb[0], r.nb_logits, atol=BF16_TOL * 8, rtol=0)
        np.testing.assert_allclose(mb[0], r.mb_logits, atol=BF16_TOL * 8, rtol=0)
        assert out[0] == r.emitted
        st = ctx.state(0)
        assert (st["t"], st["K"]) == (dec.t, dec.K)
    ctx.close()
