"""The seeded synthetic inputs (CPU): the text and weight distributions the workloads state."""
import numpy as np

from synth import TINY, WORKLOADS, make_weights, prompt, prompts, words_text, zipf_text
from synth.data import lexicon


def _words(text):
    return [w for w in text.split(b" ") if w]


def test_words_text_lengths_letters_and_determinism():
    t = words_text(0, 4096)
    assert len(t) == 4096 and t == words_text(0, 4096) and t != words_text(1, 4096)
    assert b"  " not in t and set(t) <= set(b"abcdefghijklmnopqrstuvwxyz ")
    lens = [len(w) for w in _words(t)[:-1]]           # the last word may be cut
    assert min(lens) == 1 and max(lens) == 10
    assert abs(np.mean(lens) - 5.5) < 0.3             # uniform 1..10
    assert words_text(0, 100) == t[:100]               # a shorter prompt is a prefix


def test_lexicon_and_zipf_text():
    lex = lexicon()
    assert len(lex) == 5000 and len(set(lex)) == 5000
    assert min(map(len, lex)) == 1 and max(map(len, lex)) == 12
    t = zipf_text(0, 200_000)
    assert len(t) == 200_000 and t == zipf_text(0, 200_000)
    words = _words(t)[:-1]
    rank = {w: i + 1 for i, w in enumerate(lex)}
    assert all(w in rank for w in words)
    # rank frequencies follow r^-1.1: the top ranks' observed shares against the law
    counts = np.bincount([rank[w] for w in words], minlength=5001)[1:]
    p = np.arange(1, 5001, dtype=np.float64) ** -1.1
    p /= p.sum()
    n = len(words)
    for r in (1, 2, 3, 10):
        assert abs(counts[r - 1] / n - p[r - 1]) < 4 * np.sqrt(p[r - 1] / n) + 1e-3
    # mean patch length (word plus its space): the Zipf-weighted mean over the lexicon (8.5 bytes)
    want = float(np.dot(p, [len(w) + 1 for w in lex]))
    got = float(np.mean([len(w) + 1 for w in words]))
    assert abs(want - 8.5) < 0.1 and abs(got - want) < 0.05


def test_workload_prompts_have_the_stated_shapes():
    for name, w in WORKLOADS.items():
        P = prompts(w, seqs=[0, 1])
        assert all(len(p) == w.prompt_len for p in P), name
        assert P[0] != P[1]
        assert prompt(w, 1) == P[1]


def test_weights_are_seeded_normal_with_unit_gains():
    W = make_weights(TINY)
    assert np.array_equal(W["enc.0.wq"], make_weights(TINY)["enc.0.wq"])
    big = np.concatenate([W[k].ravel() for k in W if k.endswith(("wq", "w1", "w2", "embed"))])
    assert abs(big.std() - 0.02) < 0.0005 and abs(big.mean()) < 0.0005
    for k in W:
        if k.endswith("norm"):
            assert np.all(W[k] == 1.0), k
    assert W["enc.0.w1"].shape == (TINY.d_ff, TINY.d_model)   # linear weights are [out, in]
    assert W["enc.0.w2"].shape == (TINY.d_model, TINY.d_ff)
