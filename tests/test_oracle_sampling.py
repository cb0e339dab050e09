"""Pins of the oracle's stochastic decoding (``oracle/sampling.py``) on the CPU.

The generator is checked against numpy's own Philox-4x64-10 and against the published
known-answer vectors of Philox-4x32-10; the sampling distribution against closed forms; one
speculative accept / resample round against the target distribution by quadrature over its three
uniforms; and the sampled decoders against the greedy ones in the limits where they coincide and
against plain sampling by counting.
"""
import os

import numpy as np
import pytest
from scipy import stats
from scipy.special import softmax

from oracle import model as om
from oracle.decode import SPEC, THRESH, generate_incremental, generate_reference
from oracle.sampling import (ACCEPT, DRAFT, NEXT, Sampling, draw, philox4, residual_dist,
                             sample_index, sampling_dist, spec_keep, uniform24)
from synth import make_weights
from synth.configs import ModelConfig

MICRO = ModelConfig(d_model=16, n_heads=2, head_dim=8, d_ff=64,
                    n_enc=1, n_lm=1, n_nb=1, n_mb=2, dtype="f32")
PROMPT = b"the cat sat on a mat and "


def micro_model(gain=1.0):
    return om.Model(MICRO, make_weights(MICRO, gain=gain, seed=3))


# ----------------------------------------------------------------------------- generator
@pytest.mark.parametrize("key,ctr", [((1, 2), (5, 0, 0, 0)),
                                     ((0x0123456789ABCDEF, 0xFEDCBA9876543210), (9, 3, 7, 1)),
                                     ((7, 0), (2 ** 64 - 1, 5, 0, 0))])
def test_philox4x64_matches_numpy(key, ctr):
    """numpy's Philox is Philox-4x64-10; it advances the counter (with carry) before each block."""
    g = np.random.Philox(key=np.array(key, dtype=np.uint64), counter=np.array(ctr, dtype=np.uint64))
    raw = [int(v) for v in g.random_raw(12)]
    c = list(ctr)
    want = []
    for _ in range(3):
        c[0] += 1
        for i in range(3):  # carry into the higher counter words
            if c[i] == 2 ** 64:
                c[i] = 0
                c[i + 1] += 1
        want += list(philox4(c, key, width=64))
    assert raw == want


def _kat():
    """Known-answer vectors of Philox-4x32-10 published with the generator (tests/golden)."""
    path = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")
    rows = []
    for line in open(path):
        if line.strip() and not line.startswith("#"):
            w = [int(v, 16) for v in line.split()]
            rows.append((tuple(w[0:4]), tuple(w[4:6]), tuple(w[6:10])))
    return rows


PHILOX4x32_KAT = _kat()


@pytest.mark.parametrize("ctr,key,out", PHILOX4x32_KAT)
def test_philox4x32_known_answers(ctr, key, out):
    assert philox4(ctr, key) == out


def test_uniform24_grid():
    assert uniform24(0) == 0.0
    assert uniform24(0xFF) == 0.0
    assert uniform24(0x100) == 2.0 ** -24
    assert uniform24(0x80000000) == 0.5
    assert uniform24(0xFFFFFFFF) == 1.0 - 2.0 ** -24


def test_draws_are_uniform_and_keyed_by_every_counter_word():
    u = np.array([draw(11, t, b, k, w) for t in range(40) for b in range(4) for k in (DRAFT, ACCEPT, NEXT)
                  for w in range(6)])
    assert len(np.unique(u)) == len(u)
    assert stats.kstest(u, "uniform").pvalue > 1e-3
    # the seed's high word is part of the key
    assert draw(5, 10, 0, DRAFT, 0) != draw(5 + 2 ** 32, 10, 0, DRAFT, 0)
    # words 0..3 share one block, word 4 starts the next
    assert draw(5, 10, 0, DRAFT, 4) == uniform24(philox4((10, 0, DRAFT, 1), (5, 0))[0])


# ----------------------------------------------------------------------------- distributions
def test_sampling_dist_temperature_closed_forms():
    p = np.array([0.125, 0.5, 0.125, 0.25])
    l = np.log(p) + 3.0
    np.testing.assert_allclose(sampling_dist(l, 1.0), softmax(l), rtol=1e-14)
    np.testing.assert_allclose(sampling_dist(l, 1.0), p, rtol=1e-14)
    # T = 1/2 squares the probabilities before renormalising
    np.testing.assert_allclose(sampling_dist(l, 0.5), p ** 2 / (p ** 2).sum(), rtol=1e-13)
    # T = 0 is greedy with the lowest index among equal maxima
    assert list(sampling_dist([1.0, 3.0, 3.0, 0.0], 0.0)) == [0.0, 1.0, 0.0, 0.0]


def test_sampling_dist_top_p_nucleus():
    p = np.array([0.125, 0.5, 0.125, 0.25])
    l = np.log(p)
    # order 1, 3, then 0 before 2 (equal mass, lower byte first); keep while the mass before < top_p
    np.testing.assert_allclose(sampling_dist(l, 1.0, 0.6), [0, 2 / 3, 0, 1 / 3], atol=1e-15)
    np.testing.assert_allclose(sampling_dist(l, 1.0, 0.8), [1 / 7, 4 / 7, 0, 2 / 7], atol=1e-15)
    np.testing.assert_allclose(sampling_dist(l, 1.0, 0.4), [0, 1, 0, 0], atol=1e-15)
    np.testing.assert_allclose(sampling_dist(l, 1.0, 1.0), p, rtol=1e-14)
    # the nucleus is taken after the temperature: at T = 1/2 byte 1 holds 16/22 > 0.7
    np.testing.assert_allclose(sampling_dist(l, 0.5, 0.7), [0, 1, 0, 0], atol=1e-15)


def test_sample_index_is_the_inverse_cdf_in_byte_order():
    p = np.array([0.25, 0.0, 0.5, 0.25])
    assert [sample_index(p, u) for u in (0.0, 0.2499, 0.25, 0.7499, 0.75, 1 - 2 ** -24)] == [0, 0, 2, 2, 3, 3]
    N = 4096
    f = np.bincount([sample_index(p, (k + 0.5) / N) for k in range(N)], minlength=4) / N
    np.testing.assert_allclose(f, p, atol=1.0 / N)


def test_residual_dist_closed_form():
    p = np.array([0.5, 0.25, 0.25, 0.0])
    q = np.array([0.25, 0.5, 0.0, 0.25])
    np.testing.assert_allclose(residual_dist(p, q), [0.5, 0.0, 0.5, 0.0], atol=1e-15)
    np.testing.assert_allclose(residual_dist(p, p), p)


def _pairs():
    rng = np.random.default_rng(7)
    out = []
    for k in range(6):
        lp, lq = rng.normal(0, 1.5, 6), rng.normal(0, 1.5, 6)
        T, tp = (1.0, 1.0) if k < 3 else (0.7, 0.9)
        out.append((sampling_dist(lp, T, tp), sampling_dist(lq, T, tp)))
    return out


@pytest.mark.parametrize("pq", _pairs())
def test_speculative_round_emits_the_target_distribution(pq):
    """One round: draw d from q, keep it by spec_keep, else draw from the residual. By quadrature
    over the three uniforms the emitted byte is distributed as p (to the grid's resolution), which
    fails for a ratio taken the wrong way up, a residual of q - p or one not renormalised."""
    p, q = pq
    V, N = len(p), 2048
    grid = (np.arange(N) + 0.5) / N
    f_draft = np.bincount([sample_index(q, u) for u in grid], minlength=V) / N
    r = residual_dist(p, q)
    f_res = np.bincount([sample_index(r, u) for u in grid], minlength=V) / N
    out = np.zeros(V)
    for d in range(V):
        if f_draft[d] == 0:
            continue
        keep = np.mean([spec_keep(p, q, d, u) for u in grid])
        out[d] += f_draft[d] * keep
        out += f_draft[d] * (1 - keep) * f_res
    np.testing.assert_allclose(out, p, atol=3.0 * V / N)


# ----------------------------------------------------------------------------- decode loops
@pytest.mark.parametrize("mode", [SPEC, THRESH])
@pytest.mark.parametrize("samp", [Sampling(1e-4, 1.0, 3), Sampling(1.0, 1e-9, 4)])
def test_sampled_decoding_reduces_to_greedy(mode, samp):
    """As T -> 0, or with a nucleus of one byte, every sampling distribution is the argmax: the
    sampled decoder must then emit the greedy decoder's bytes with the same accepted counts."""
    M = micro_model(gain=40.0)
    want, rw = generate_reference(M, PROMPT, 4, 0.6, mode, 24)
    got, rg = generate_reference(M, PROMPT, 4, 0.6, mode, 24, samp=samp)
    assert got == want
    assert [r.a for r in rg] == [r.a for r in rw]
    assert sum(r.a for r in rw) > 0


@pytest.mark.parametrize("mode,tau,gain", [(SPEC, 0.75, 8.0), (THRESH, 0.15, 20.0)])
def test_sampled_incremental_equals_full_recompute(mode, tau, gain):
    M = micro_model(gain=gain)
    samp = Sampling(0.7, 0.9, 12345)
    out_r, rr = generate_reference(M, PROMPT, 4, tau, mode, 30, samp=samp, b=2)
    out_i, ri = generate_incremental(M, PROMPT, 4, tau, mode, 30, samp=samp, b=2)
    assert out_r == out_i
    assert [(r.c1, r.drafts, r.a) for r in rr] == [(r.c1, r.drafts, r.a) for r in ri]
    assert 0 < sum(r.a for r in rr) < 3 * len(rr)
    # another sequence index draws other numbers
    assert generate_reference(M, PROMPT, 4, tau, mode, 30, samp=samp, b=3)[0] != out_r


def test_speculative_sampling_matches_plain_sampling():
    """Counting over seeds: the first two bytes of speculative sampling follow the plain sampling
    distribution P(x1) P(x2 | x1), computed from full forwards (chi-square, expected counts >= 5)."""
    M = micro_model(gain=20.0)
    T, tp = 0.7, 0.9
    t = len(PROMPT)
    p1 = sampling_dist(om.forward_full(M, PROMPT).nb_logits[t - 1], T, tp)
    joint = {}
    for x1 in np.nonzero(p1)[0]:
        p2 = sampling_dist(om.forward_full(M, PROMPT + bytes([x1])).nb_logits[t], T, tp)
        for x2 in np.nonzero(p2)[0]:
            joint[(int(x1), int(x2))] = p1[x1] * p2[x2]
    S = 3000
    seen = {}
    accepted = 0
    for s in range(S):
        out, recs = generate_reference(M, PROMPT, 3, 0.75, SPEC, 2, samp=Sampling(T, tp, 1000 + s))
        key = (out[0], out[1])
        assert key in joint
        seen[key] = seen.get(key, 0) + 1
        accepted += recs[0].a
    assert 0.1 * S < accepted < 1.5 * S  # drafts are kept and rejected
    keys = sorted(joint, key=lambda k: -joint[k])
    big = [k for k in keys if joint[k] * S >= 5]
    obs = [seen.get(k, 0) for k in big] + [S - sum(seen.get(k, 0) for k in big)]
    exp = [joint[k] * S for k in big] + [S * (1 - sum(joint[k] for k in big))]
    assert len(big) >= 4
    assert stats.chisquare(obs, exp).pvalue > 1e-3


@pytest.mark.parametrize("pq", _pairs())
def test_speculative_acceptance_rate_is_the_overlap(pq):
    """The probability that a draft drawn from q is kept is sum_x min(p(x), q(x)) (the expected
    acceptance rate of speculative sampling), by quadrature over the draft's and the test's
    uniforms."""
    p, q = pq
    N = 2048
    grid = (np.arange(N) + 0.5) / N
    kept = 0.0
    for ud in grid:
        d = sample_index(q, ud)
        kept += np.mean([spec_keep(p, q, d, ua) for ua in grid[::4]])
    np.testing.assert_allclose(kept / N, np.minimum(p, q).sum(), atol=3.0 * len(p) / N)


def test_n1_sampling_is_plain_sampling():
    """With n = 1 there are no drafts: every step draws one byte from the next-byte sampling
    distribution with the step's NEXT uniform (c_1 of the step that starts at length t)."""
    M = micro_model(gain=8.0)
    samp = Sampling(0.7, 0.9, 77)
    x = bytearray(PROMPT)
    for _ in range(10):
        p = sampling_dist(om.forward_full(M, x).nb_logits[-1], samp.temperature, samp.top_p)
        x.append(sample_index(p, draw(samp.seed, len(x), 0, NEXT, 0)))
    want = bytes(x[len(PROMPT):])
    for mode in (THRESH, SPEC):
        assert generate_reference(M, PROMPT, 1, 0.75, mode, 10, samp=samp)[0] == want
        assert generate_incremental(M, PROMPT, 1, 0.75, mode, 10, samp=samp)[0] == want
