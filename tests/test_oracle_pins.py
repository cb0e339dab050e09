"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every test here runs on the CPU. Each targets a plausible mistake in the oracle
(a dropped term, a wrong sign or index, a transposed operand, an off-by-one in the
segment/latent alignment) through a closed form, a special case that reduces to a
textbook computation, an invariant the paper states, or brute force on tiny inputs.
"""
import math

import numpy as np
import pytest
from scipy.special import expit

from oracle import model as om
from oracle.decode import (SPEC, THRESH, IncrementalDecoder, generate_incremental,
                           generate_reference, greedy_decode)
from synth import TINY, make_weights, param_count, PAPER, words_text
from synth.configs import ModelConfig

MICRO = ModelConfig(d_model=16, n_heads=2, head_dim=8, d_ff=64,
                    n_enc=1, n_lm=1, n_nb=1, n_mb=2, dtype="f32")


def micro_model(gain=1.0, **kw):
    cfg = MICRO.replace(**kw)
    return om.Model(cfg, make_weights(cfg, gain=gain, seed=3))


# ----------------------------------------------------------------------------- block math
def test_rmsnorm_closed_form():
    c, eps = -1.7, 1e-6
    g = np.linspace(0.5, 2.0, 8)
    got = om.rmsnorm(np.full(8, c), g, eps)
    np.testing.assert_allclose(got, c / math.sqrt(c * c + eps) * g, rtol=1e-14)
    # unit-RMS input with eps = 0 passes through unchanged
    x = np.array([1.0, -1.0, 1.0, -1.0])
    np.testing.assert_allclose(om.rmsnorm(x, np.ones(4), 0.0), x, rtol=1e-15)


def test_silu_matches_library_sigmoid():
    x = np.linspace(-30, 30, 601)
    np.testing.assert_allclose(om.silu(x), x * expit(x), rtol=1e-12, atol=1e-300)
    assert om.silu(np.array([0.0]))[0] == 0.0


def test_rope_is_a_plane_rotation_per_pair():
    base = 1e5
    # h_d = 2: one pair, frequency base^0 = 1, so position p rotates by p radians
    v = np.array([[[0.3, -0.8]]])
    for p in (0, 1, 5, 17):
        got = om.rope(v, np.array([p]), base)[0, 0]
        R = np.array([[math.cos(p), -math.sin(p)], [math.sin(p), math.cos(p)]])
        np.testing.assert_allclose(got, R @ v[0, 0], rtol=1e-12, atol=1e-15)
    # pair i of h_d = 8 turns by base^(-2i/8) per position
    hd = 8
    for i in range(hd // 2):
        e = np.zeros((1, 1, hd))
        e[0, 0, 2 * i] = 1.0
        r = om.rope(e, np.array([1]), base)[0, 0]
        ang = math.atan2(r[2 * i + 1], r[2 * i])
        assert abs(ang - base ** (-2 * i / hd)) < 1e-12
        assert abs(np.linalg.norm(r) - 1.0) < 1e-14


def test_rope_scores_depend_on_offset_only():
    rng = np.random.default_rng(1)
    q = rng.standard_normal((1, 2, 8))
    k = rng.standard_normal((1, 2, 8))
    def score(pq, pk):
        return np.sum(om.rope(q, np.array([pq]), 1e5) * om.rope(k, np.array([pk]), 1e5))
    s0 = score(9, 4)
    for shift in (1, 13, 250):
        assert abs(score(9 + shift, 4 + shift) - s0) < 1e-12


def test_attention_special_cases():
    rng = np.random.default_rng(2)
    v = rng.standard_normal((5, 1, 4))
    k = rng.standard_normal((5, 1, 4))
    # one visible key: the output is that key's value
    q = rng.standard_normal((1, 1, 4))
    mask = np.array([[False, False, True, False, False]])
    np.testing.assert_allclose(om.attend(q, k, v, mask, 0.5)[0], v[2], rtol=1e-14)
    # zero query: uniform weights, the mean of the visible values
    mask = np.array([[True, True, False, True, False]])
    np.testing.assert_allclose(om.attend(np.zeros((1, 1, 4)), k, v, mask, 0.5)[0],
                               v[[0, 1, 3]].mean(axis=0), rtol=1e-13)
    # two keys, scores 2 and 0 after scaling: weights e^2/(e^2+1), 1/(e^2+1)
    q = np.array([[[1.0, 0.0]]])
    k2 = np.array([[[4.0, 0.0]], [[0.0, 3.0]]])
    v2 = np.array([[[1.0, 0.0]], [[0.0, 1.0]]])
    out = om.attend(q, k2, v2, np.array([[True, True]]), 0.5)[0, 0]
    w = math.exp(2) / (math.exp(2) + 1)
    np.testing.assert_allclose(out, [w, 1 - w], rtol=1e-14)


def _groups_from_text(x):
    g, out = 0, []
    for c in x:
        if c == 0x20:
            g += 1
        out.append(g)
    return out


def test_lca_mask_matches_the_verbal_definition():
    """Figure 2: a query sees itself, earlier bytes of its own latent group and every
    byte of the immediately preceding group; nothing later, nothing older."""
    x = b"ab cde f  gh"
    grp = _groups_from_text(x)
    m = om.lca_mask(grp)
    for p in range(len(x)):
        members = {q for q in range(len(x)) if grp[q] == grp[p] and q <= p}
        prev = {q for q in range(len(x)) if grp[q] == grp[p] - 1}
        for q in range(len(x)):
            assert m[p, q] == (q in members or q in prev), (p, q)


def test_segments_round_trip_and_latent_index():
    for seq in range(5):
        x = words_text(seq, 97) + b"  x "
        segs = om.closed_segments(TINY, x)
        open_tail = x[segs[-1][1] + 1:] if segs else x
        joined = b"".join(x[s:e + 1] for s, e in segs) + open_tail
        assert joined == x
        for s, e in segs:
            assert x[e] == 0x20 and x[s:e].count(b" ") == 0
        Kp = om.latent_index(TINY, x)
        assert list(Kp) == _groups_from_text(x)
        for g in range(1, Kp[-1] + 1):
            assert om.group_start(TINY, x, g) == segs[g - 1][1]


def test_pool_is_segment_mean():
    h = np.arange(12, dtype=np.float64).reshape(6, 2)
    z = om.pool(h, [(0, 1), (2, 5)])
    np.testing.assert_allclose(z, [[1.0, 2.0], [7.0, 8.0]])


# ----------------------------------------------------------------------------- blocks
def _identity_block(cfg, **over):
    d, f = cfg.d_model, cfg.d_ff
    lw = {"attn_norm": np.ones(d), "wq": np.zeros((d, d)), "wk": np.zeros((d, d)),
          "wv": np.eye(d), "wo": np.eye(d), "mlp_norm": np.ones(d),
          "w1": np.zeros((f, d)), "w3": np.zeros((f, d)), "w2": np.zeros((d, f))}
    lw.update(over)
    return lw


def test_block_with_zero_output_projections_is_identity():
    cfg = MICRO
    rng = np.random.default_rng(4)
    lw = {k: rng.standard_normal(v.shape) for k, v in _identity_block(cfg).items()}
    lw["wo"] = np.zeros_like(lw["wo"])
    lw["w2"] = np.zeros_like(lw["w2"])
    x = rng.standard_normal((7, cfg.d_model))
    y, _, _ = om.block(cfg, lw, x, np.arange(7), om.causal_mask(0, 7))
    np.testing.assert_allclose(y, x, rtol=0, atol=0)


def test_block_uniform_attention_is_running_mean_of_normalised_rows():
    """Wq = Wk = 0 gives uniform causal weights; with Wv = Wo = I and no MLP the block
    adds to row p the mean of RMSNorm(x_q) over q <= p."""
    cfg = MICRO
    rng = np.random.default_rng(5)
    x = rng.standard_normal((6, cfg.d_model)) * 3
    y, _, _ = om.block(cfg, _identity_block(cfg), x, np.arange(6), om.causal_mask(0, 6))
    for p in range(6):
        rows = [x[q] / math.sqrt(np.mean(x[q] ** 2) + cfg.rms_eps) for q in range(p + 1)]
        np.testing.assert_allclose(y[p], x[p] + np.mean(rows, axis=0), rtol=1e-12)


def test_block_mlp_is_swiglu_w2_silu_w1_times_w3():
    cfg = MICRO.replace(d_ff=3)
    d = cfg.d_model
    rng = np.random.default_rng(6)
    w1, w3, w2 = rng.standard_normal((3, d)), rng.standard_normal((3, d)), rng.standard_normal((d, 3))
    lw = _identity_block(cfg, wo=np.zeros((d, d)), w1=w1, w3=w3, w2=w2)
    x = rng.standard_normal((1, d))
    y, _, _ = om.block(cfg, lw, x, np.arange(1), om.causal_mask(0, 1))
    m = x[0] / math.sqrt(np.mean(x[0] ** 2) + cfg.rms_eps)
    a, b = w1 @ m, w3 @ m
    want = x[0] + sum(w2[:, j] * (a[j] * expit(a[j]) * b[j]) for j in range(3))
    np.testing.assert_allclose(y[0], want, rtol=1e-12)


# ----------------------------------------------------------------------------- wiring
def _zero_layer_model(seed=8):
    cfg = MICRO.replace(n_enc=0, n_lm=0, n_nb=0, n_mb=0)
    return om.Model(cfg, make_weights(cfg, seed=seed))


def test_zero_layer_next_byte_logits_use_the_latent_of_the_closing_segment():
    """With empty stacks h_e = E[x], o = u = [BOS, z_1..]; byte p is decoded from
    o_{K(p)} + E[x_p], where a boundary byte already sees the mean of its own segment
    and any other byte sees the latent of the segment before its own."""
    M = _zero_layer_model()
    W = M.w
    x = b"ab cd e"
    F = om.forward_full(M, x)
    E = W["embed"]
    seg1 = (E[ord("a")] + E[ord("b")] + E[0x20]) / 3
    seg2 = (E[ord("c")] + E[ord("d")] + E[0x20]) / 3
    latent_for = [W["lm.bos"], W["lm.bos"], seg1, seg1, seg1, seg2, seg2]
    for p, c in enumerate(x):
        h = latent_for[p] + E[c]
        want = W["unembed"] @ (h / math.sqrt(np.mean(h * h) + M.cfg.rms_eps))
        np.testing.assert_allclose(F.nb_logits[p], want, rtol=1e-12, atol=1e-14)


def test_zero_layer_mb_input_adds_r2_before_upsampling():
    """With empty stacks every draft row of group g decodes o_g + u_g = 2 u_g, whose
    RMSNorm equals that of u_g (Algorithm 1, drafting input)."""
    M = _zero_layer_model()
    x = b"ab cd ef"
    F = om.forward_full(M, x)
    lg = om.mb_draft_logits(M, F.Kp, F.o, F.u, len(x), 4, x)
    u = F.u[2]
    want = M.w["unembed"] @ (u / math.sqrt(np.mean(u * u) + M.cfg.rms_eps / 4))
    for r in lg:
        np.testing.assert_allclose(r, want, rtol=1e-12, atol=1e-14)


def test_window_is_previous_plus_current_group_with_duplicates():
    cfg = TINY
    x = b"abc de fgh"
    Kp = om.latent_index(cfg, x)
    o = u = np.arange(3 * 2, dtype=np.float64).reshape(3, 2)
    m, pos, grp = om.window_draft_inputs(cfg, Kp, o, u, len(x), 5, x)
    # current group 2 starts at the second space (pos 6); previous group 1 at pos 3
    assert list(pos) == [3, 4, 5, 6, 7, 8, 9, 10, 11, 12]
    assert list(grp) == [1, 1, 1, 2, 2, 2, 2, 2, 2, 2]
    np.testing.assert_allclose(m[0], o[1] + u[1])
    np.testing.assert_allclose(m[-1], o[2] + u[2])
    # group 0 has no predecessor: the window starts at byte 0
    x0 = b"abcd"
    m, pos, grp = om.window_draft_inputs(cfg, om.latent_index(cfg, x0), o, u, 4, 3, x0)
    assert list(pos) == [0, 1, 2, 3, 4] and list(grp) == [0] * 5


def test_lca_inside_the_window_is_plain_causal():
    grp = [3, 3, 3, 4, 4, 4, 4]
    np.testing.assert_array_equal(om.lca_mask(grp), om.causal_mask(0, len(grp)))


def test_one_layer_window_equals_full_sequence_lca_forward():
    """With one MB layer the window slice of Algorithm 1 loses nothing: the LCA mask
    already hides everything before the previous group."""
    M = micro_model(n_mb=1)
    x = b"ab cde fg hij k"
    F = om.forward_full(M, x)
    for n in (2, 3, 5):
        w = om.mb_draft_logits(M, F.Kp, F.o, F.u, len(x), n, x)
        full = om.full_sequence_lca_logits(M, F.Kp, F.o, F.u, extra=n - 2)
        np.testing.assert_allclose(w, full[-(n - 1):], rtol=1e-10, atol=1e-12)


# ----------------------------------------------------------------------------- causality
def test_next_byte_logits_are_causal():
    M = micro_model()
    x = bytearray(b"ab cd efg hi jk")
    F = om.forward_full(M, bytes(x))
    for q in (4, 8, 14):
        y = bytearray(x)
        y[q] = ord("z") if y[q] != ord("z") else ord("y")
        G = om.forward_full(M, bytes(y))
        np.testing.assert_allclose(G.nb_logits[:q], F.nb_logits[:q], rtol=1e-12, atol=1e-13)
        assert np.abs(G.nb_logits[q:] - F.nb_logits[q:]).max() > 1e-9


def test_bos_shift_keeps_latents_causal():
    M = micro_model()
    x = b"ab cd efg hi "
    F = om.forward_full(M, x)
    y = b"ab cd exg hi "     # changes segment 3 only
    G = om.forward_full(M, y)
    np.testing.assert_allclose(G.o[:3], F.o[:3], rtol=1e-12, atol=1e-13)
    assert np.abs(G.o[3] - F.o[3]).max() > 1e-9


def test_mb_draft_ignores_bytes_of_the_current_group():
    """Section 3: drafts of a group depend only on bytes up to the boundary that opened
    it, so changing non-boundary bytes after it leaves them unchanged."""
    M = micro_model()
    x = b"ab cd efgh"
    F = om.forward_full(M, x)
    base = om.mb_draft_logits(M, F.Kp, F.o, F.u, len(x), 4, x)
    y = b"ab cd xyzw"
    G = om.forward_full(M, y)
    got = om.mb_draft_logits(M, G.Kp, G.o, G.u, len(y), 4, y)
    np.testing.assert_allclose(got, base, rtol=1e-12, atol=1e-13)
    z = b"ab cx efgh"       # a byte of the previous group does matter
    H = om.forward_full(M, z)
    assert np.abs(om.mb_draft_logits(M, H.Kp, H.o, H.u, len(z), 4, z) - base).max() > 1e-9


# ----------------------------------------------------------------------------- decode loop
PROMPT = b"the cat sat on a mat and "


def test_n1_is_greedy_next_byte_decoding():
    M = micro_model()
    want = greedy_decode(M, PROMPT, 12)
    got, recs = generate_reference(M, PROMPT, 1, 0.75, THRESH, 12)
    assert got == want and all(len(r.emitted) == 1 for r in recs)


@pytest.mark.parametrize("n", [2, 3, 5])
def test_spec_acceptance_reproduces_greedy(n):
    """Section 6.2: speculative acceptance makes the output equal next-byte decoding."""
    M = micro_model(gain=40.0)
    want = greedy_decode(M, PROMPT, 14)
    got, recs = generate_reference(M, PROMPT, n, 0.75, SPEC, 14)
    assert got == want
    assert sum(r.a for r in recs) > 0


def test_threshold_extremes():
    M = micro_model(gain=40.0)
    want = greedy_decode(M, PROMPT, 10)
    got, recs = generate_reference(M, PROMPT, 4, 1.5, THRESH, 10)
    assert got == want and all(r.a == 0 for r in recs)
    got, recs = generate_reference(M, PROMPT, 4, 0.0, THRESH, 10)
    assert [len(r.emitted) for r in recs] == [4, 4, 2]


def test_accepted_drafts_form_a_prefix_of_passing_probabilities():
    M = micro_model(gain=40.0)
    _, recs = generate_reference(M, PROMPT, 5, 0.6, THRESH, 30)
    for r in recs:
        assert 0 <= r.a <= 4
        assert all(p >= 0.6 for p in r.probs[:r.a])
        if r.a < 4:
            assert r.probs[r.a] < 0.6


CASES = [
    dict(n=3, tau=0.75, mode=THRESH, gain=1.0),
    dict(n=4, tau=0.5, mode=THRESH, gain=40.0),
    dict(n=5, tau=0.75, mode=SPEC, gain=40.0),
]


@pytest.mark.parametrize("case", CASES)
def test_incremental_equals_full_recompute(case):
    M = micro_model(gain=case["gain"])
    out_r, rr = generate_reference(M, PROMPT, case["n"], case["tau"], case["mode"], 20,
                                   record_nb=True)
    out_i, ri = generate_incremental(M, PROMPT, case["n"], case["tau"], case["mode"], 20)
    assert out_r == out_i
    for a, b in zip(rr, ri):
        assert (a.c1, a.drafts, a.a, a.emitted, a.t, a.K) == (b.c1, b.drafts, b.a, b.emitted, b.t, b.K)
        np.testing.assert_allclose(b.mb_logits, a.mb_logits, rtol=1e-9, atol=1e-11)
        np.testing.assert_allclose(b.nb_logits, a.nb_logits, rtol=1e-9, atol=1e-11)


def test_incremental_rollback_across_forced_boundaries():
    """Candidates holding boundaries, with every accepted count, exercise the LM module
    on speculative segments and the rollback of the rejected ones."""
    M = micro_model()
    pats = [b"ab c", b" abc", b"a  b", b"    ", b"abcd", b"x y ", b"  xy"]
    force = [0, 3, 1, 2, 3, 0, 2, 1, 3]
    fc = lambda s: pats[s % len(pats)]
    out_r, rr = generate_reference(M, PROMPT, 4, 0.75, THRESH, 40, force=force,
                                   record_nb=True, force_cand=fc)
    out_i, ri = generate_incremental(M, PROMPT, 4, 0.75, THRESH, 40, force=force, force_cand=fc)
    assert out_r == out_i
    assert out_r.count(b" ") >= 8
    for a, b in zip(rr, ri):
        assert (a.t, a.K) == (b.t, b.K)
        np.testing.assert_allclose(b.mb_logits, a.mb_logits, rtol=1e-9, atol=1e-11)
        np.testing.assert_allclose(b.nb_logits, a.nb_logits, rtol=1e-9, atol=1e-11)


def test_mlp_head_drafts():
    """MLP-MBP (Section 4.1): head j decodes the last next-byte hidden state through
    its residual SiLU layers; heads are independent of each other and of n."""
    cfg = MICRO.replace(mb_kind="mlp", n_mb=3, n_mlp_heads=4)
    M = om.Model(cfg, make_weights(cfg, seed=5))
    F = om.forward_full(M, PROMPT)
    l5 = om.mb_draft_logits(M, F.Kp, F.o, F.u, len(PROMPT), 5, PROMPT, y_last=F.y[-1])
    l3 = om.mb_draft_logits(M, F.Kp, F.o, F.u, len(PROMPT), 3, PROMPT, y_last=F.y[-1])
    np.testing.assert_allclose(l5[:2], l3, rtol=1e-14)
    v = F.y[-1].copy()
    for l in range(3):
        a = M.w[f"mlp.1.{l}.w"] @ v
        v = v + a * expit(a)
    want = M.w["unembed"] @ (v / math.sqrt(np.mean(v * v) + cfg.rms_eps))
    np.testing.assert_allclose(l5[1], want, rtol=1e-11, atol=1e-13)
    out_r, _ = generate_reference(M, PROMPT, 5, 0.5, THRESH, 12)
    out_i, _ = generate_incremental(M, PROMPT, 5, 0.5, THRESH, 12)
    assert out_r == out_i


def test_paper_parameter_count():
    """Section 4.3 states 373M parameters for the 2/16/2/2 split at d = 1024 and inner
    size 4096 (Section 4.2); the SwiGLU-4d block gives 369.7M, within 1%."""
    n = param_count(PAPER)
    assert abs(n - 373e6) / 373e6 < 0.01
    assert n == 22 * 16 * 1024 ** 2 + 2 * 256 * 1024 + (2 * 22 + 3) * 1024


def test_head_decisions_ties_and_probability():
    """Reading R12 (argmax takes the lowest byte among equal maxima) and R4 (the drafter's
    probability of its argmax, exp(l_max - logsumexp))."""
    from oracle.model import greedy, max_prob
    lg = np.zeros(256)
    assert greedy(lg) == 0 and abs(max_prob(lg, 0) - 1 / 256) < 1e-15
    lg[[7, 200]] = 3.0
    assert greedy(lg) == 7
    p = max_prob(lg, 7)
    assert abs(p - np.e ** 3 / (2 * np.e ** 3 + 254)) < 1e-14
    big = lg + 1e4  # a common offset changes nothing and does not overflow
    assert greedy(big) == 7 and abs(max_prob(big, 7) - p) < 1e-12


def test_learned_predictor_that_fires_on_spaces_is_the_space_rule():
    """A predictor that reads a space marker of the embedding, behind an encoder whose output
    projections are zero (so h_e = embedding), must segment, pool, draft and decode exactly as the
    space rule does, through the cached decoder's rollbacks as well."""
    cfg_l = MICRO.replace(boundary="learned", d_bp=1)
    W = make_weights(cfg_l, gain=40.0, seed=3)
    W["embed"][:, 0] = 0.0
    W["embed"][0x20, 0] = 4.0
    W["enc.0.wo"][:] = 0.0
    W["enc.0.w2"][:] = 0.0
    W["bp.w1"][:] = 0.0
    W["bp.w1"][0, 0] = 1.0
    W["bp.w2"][:] = 1.0
    W["bp.bias"][:] = -1.0  # SiLU(4) - 1 > 0 on a space, SiLU(0) - 1 < 0 elsewhere
    ML, MS = om.Model(cfg_l, W), om.Model(MICRO, W)
    x = b"ab cd  efg h"
    FL, FS = om.forward_full(ML, x), om.forward_full(MS, x)
    assert list(FL.b) == [c == 0x20 for c in x]
    np.testing.assert_array_equal(FL.nb_logits, FS.nb_logits)
    pats = [b"ab c", b" abc", b"a  b", b"abcd", b"x y "]
    fc = lambda s: pats[s % len(pats)]  # noqa: E731
    for mode in (THRESH, SPEC):
        want, rw = generate_incremental(MS, PROMPT, 4, 0.6, mode, 24, force_cand=fc)
        got, rg = generate_incremental(ML, PROMPT, 4, 0.6, mode, 24, force_cand=fc)
        assert got == want
        assert [(r.a, r.t, r.K) for r in rg] == [(r.a, r.t, r.K) for r in rw]
        ref, rr = generate_reference(ML, PROMPT, 4, 0.6, mode, 24, force_cand=fc)
        assert ref == want and [r.K for r in rr] == [r.K for r in rw]


def test_incremental_equals_full_recompute_at_paper_size():
    """The cached decoder against the full recompute on the paper-size model (2/16/2/2 blocks,
    d = 1024, 16 heads of 64, the calibrated gains of the batch-1 workload) over a short prompt:
    shapes that the micro models do not reach (16 heads, 16 LM blocks, bf16-rounded weights)."""
    from synth import WORKLOADS, cached_weights, prompt, weight_gains
    w = WORKLOADS["paper_b1"]
    M = om.Model(w.model, cached_weights(w.model, **weight_gains(w, True)))
    p = prompt(w, 0, 96)
    out_r, rr = generate_reference(M, p, 3, 0.75, THRESH, 6, record_nb=True)
    out_i, ri = generate_incremental(M, p, 3, 0.75, THRESH, 6)
    assert out_r == out_i
    for a, b in zip(rr, ri):
        assert (a.c1, a.drafts, a.a, a.t, a.K) == (b.c1, b.drafts, b.a, b.t, b.K)
        np.testing.assert_allclose(b.mb_logits, a.mb_logits, rtol=1e-8, atol=1e-8)
        np.testing.assert_allclose(b.nb_logits, a.nb_logits, rtol=1e-8, atol=1e-8)
    assert p.count(b" ") >= 5  # the prompt has closed segments for the LM module
