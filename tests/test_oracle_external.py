"""Pins of the oracle's external verification (``oracle/external.py``) on the CPU.

Section 6.3: verifying the LCA model's drafts with an external model gives that model's own
output. So the committed bytes must be the verifier's greedy decoding whatever the drafts are;
with the drafter as its own verifier the loop must be the self-speculative one of Section 6.2;
and the cached form must equal the full recompute, segments closed by rejected candidates included.
"""
import numpy as np
import pytest

from oracle import model as om
from oracle.decode import SPEC, generate_reference, greedy_decode
from oracle.external import acceptance_rate, generate_external, generate_external_reference
from synth import make_weights
from synth.configs import ModelConfig

MICRO = ModelConfig(d_model=16, n_heads=2, head_dim=8, d_ff=64,
                    n_enc=1, n_lm=1, n_nb=1, n_mb=2, dtype="f32")
# the verifier's shape: a learned boundary predictor, a deeper next-byte decoder, no multi-byte head
FXT = MICRO.replace(boundary="learned", d_bp=8, n_nb=2, n_mb=0)
PROMPT = b"the cat sat on a mat and "


@pytest.fixture(scope="module")
def drafter():
    return om.Model(MICRO, make_weights(MICRO, gain=40.0, seed=3))


@pytest.fixture(scope="module")
def verifier():
    """FxT-shaped, its predictor's bias at the upper quartile of its logits over the prompt."""
    V = om.Model(FXT, make_weights(FXT, gain=40.0, seed=11))
    h = om.forward_full(V, PROMPT).h_e
    lg = om.boundary_logits(V, h) - V.w["bp.bias"][0]
    V.w["bp.bias"][0] = -np.quantile(lg, 0.75)
    return V


def test_self_verification_is_the_speculative_loop(drafter):
    want, rw = generate_reference(drafter, PROMPT, 4, 0.0, SPEC, 30)
    for gen in (generate_external_reference, generate_external):
        got, rg = gen(drafter, drafter, PROMPT, 4, 30)
        assert got == want
        assert [(r.a, r.t, r.K) for r in rg] == [(r.a, r.t, r.K) for r in rw]


def _hook(target, P):
    """Drafts taken from the verifier's own continuation `target`, every third one replaced by a
    space (the drafter's boundary byte), so that drafts are kept, rejected, and close segments."""
    def hook(t, drafts):
        out = []
        for i in range(len(drafts)):
            j = t - len(P) + 1 + i
            out.append(0x20 if (t + i) % 3 == 0 or j >= len(target) else target[j])
        return out
    return hook


@pytest.mark.parametrize("n", [2, 4, 6])
def test_external_output_is_the_verifiers_greedy_decoding(drafter, verifier, n):
    G = 30
    want = greedy_decode(verifier, PROMPT, G)
    assert om.forward_full(verifier, PROMPT + want).b.sum() >= 8  # the verifier segments its text
    hook = _hook(want, PROMPT)
    ref, rr = generate_external_reference(drafter, verifier, PROMPT, n, G, draft_hook=hook)
    inc, ri = generate_external(drafter, verifier, PROMPT, n, G, draft_hook=hook)
    assert ref == want and inc == want
    assert [(r.a, r.t, r.K) for r in ri] == [(r.a, r.t, r.K) for r in rr]
    for a, b in zip(rr, ri):
        np.testing.assert_allclose(b.mb_logits, a.mb_logits, rtol=1e-9, atol=1e-11)
        np.testing.assert_allclose(b.nb_logits, a.nb_logits, rtol=1e-9, atol=1e-11)
    rate = acceptance_rate(rr, n)
    assert 0.0 < rate < 1.0
    # unhooked, the drafter's own drafts: the output is still the verifier's
    assert generate_external(drafter, verifier, PROMPT, n, 12)[0] == want[:12]
