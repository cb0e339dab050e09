"""Brute-force pin of the oracle's whole model and decode loop (CPU).

The chain of Section 2.2, Section 3 and Algorithm 1, written here as scalar loops over explicit
indices on a tiny model with random weights (d = 8, two heads, T <= 40 bytes), with no call into
``oracle/``; the oracle's vectorised ``forward_full``, ``mb_draft_logits``, ``generate_reference``
and ``IncrementalDecoder`` must agree with it:

  e_p    = E[x_p]
  h_e    = encoder blocks over e (causal, RoPE at byte position p)
  b_p    = [x_p == 0x20], or with the learned predictor [sum_j w2_j SiLU(sum_c W1_jc h_e[p]_c) + c0 > 0];
           K(p) = #{q <= p : b_q}; closed segment k = bytes after the (k-1)-th boundary up to and
           including the k-th
  z_k    = mean of h_e over segment k;  u_0 = BOS, u_k = z_k
  o      = LM blocks over u_0..u_K (causal, RoPE at latent index)
  y_p    = next-byte blocks over o_{K(p)} + h_e[p] (causal, RoPE p); logits_p = W_u RMSNorm_nb(y_p)
  window = the committed positions q < t with K(q) >= K(t-1) - 1, then n-2 copies at t..t+n-3 in
           group K(t-1); input row = o_g + u_g of its group g; multi-byte blocks where row i sees
           row j iff j <= i and g_j in {g_i, g_i - 1}; the last n-1 rows through RMSNorm_mb, W_u
  step   = c_1 = argmax of the next-byte logits at t-1; drafts = argmaxes of the window rows;
           THRESH keeps drafts while their softmax probability >= tau; SPEC while each equals the
           next-byte argmax of the row before it in a forward over the committed bytes and the
           candidates; commit 1 + a bytes.

A plausible slip in the oracle's composition (pooling over the wrong span, K(p) counted exclusively
so that the upsampled latent comes one group late, the window starting one group early, the draft
rows taken from the wrong end) changes these values and fails one of the tests below. (A constant
shift of every LM position is not such a slip: rotary scores depend only on position offsets.)"""
import math
import random

import numpy as np
import pytest

from oracle import SPEC, THRESH, IncrementalDecoder, Model, forward_full, generate_reference
from oracle.model import mb_draft_logits
from synth.configs import ModelConfig

CFG = ModelConfig(d_model=8, n_heads=2, head_dim=4, d_ff=12, n_enc=1, n_lm=2, n_nb=1, n_mb=2, dtype="f32")
CFG_MLP = CFG.replace(mb_kind="mlp", n_mb=3, n_mlp_heads=3)
CFG_BP = CFG.replace(boundary="learned", d_bp=6)
SP = 0x20


# ----------------------------------------------------------------------------- random weights
def _g(rng, scale):
    return rng.gauss(0.0, scale)


def _mat(rng, rows, cols, scale):
    return [[_g(rng, scale) for _ in range(cols)] for _ in range(rows)]


def make_weights(cfg, seed, unembed_scale=1.5):
    rng = random.Random(seed)
    d, f = cfg.d_model, cfg.d_ff
    W = {"embed": _mat(rng, 256, d, 1.0), "unembed": _mat(rng, 256, d, unembed_scale),
         "lm.bos": [_g(rng, 1.0) for _ in range(d)],
         "nb.norm": [1.0 + _g(rng, 0.2) for _ in range(d)], "mb.norm": [1.0 + _g(rng, 0.2) for _ in range(d)]}
    stacks = [("enc", cfg.n_enc), ("lm", cfg.n_lm), ("nb", cfg.n_nb)]
    if cfg.mb_kind == "lca":
        stacks.append(("mb", cfg.n_mb))
    for pre, n in stacks:
        for l in range(n):
            b = f"{pre}.{l}."
            W[b + "attn_norm"] = [1.0 + _g(rng, 0.2) for _ in range(d)]
            W[b + "mlp_norm"] = [1.0 + _g(rng, 0.2) for _ in range(d)]
            for nm in ("wq", "wk", "wv", "wo"):
                W[b + nm] = _mat(rng, d, d, 0.5)
            W[b + "w1"] = _mat(rng, f, d, 0.5)
            W[b + "w3"] = _mat(rng, f, d, 0.5)
            W[b + "w2"] = _mat(rng, d, f, 0.5)
    if cfg.mb_kind == "mlp":
        for j in range(cfg.n_mlp_heads):
            for l in range(cfg.n_mb):
                W[f"mlp.{j}.{l}.w"] = _mat(rng, d, d, 0.5)
    if cfg.boundary == "learned":
        W["bp.w1"] = _mat(rng, cfg.d_bp, d, 0.5)
        W["bp.w2"] = [_g(rng, 1.0) for _ in range(cfg.d_bp)]
        W["bp.bias"] = [0.0]
    return W


def as_model(cfg, W):
    return Model(cfg, {k: np.asarray(v, dtype=np.float64) for k, v in W.items()})


# ----------------------------------------------------------------------------- scalar definitions
def _norm(v, g, eps):
    r = 1.0 / math.sqrt(sum(e * e for e in v) / len(v) + eps)
    return [v[c] * r * g[c] for c in range(len(v))]


def _matvec(M, v):
    return [sum(M[o][c] * v[c] for c in range(len(v))) for o in range(len(M))]


def _rope(cfg, v, pos):
    out = list(v)
    hd = cfg.head_dim
    for h in range(cfg.n_heads):
        for i in range(hd // 2):
            th = pos * cfg.rope_base ** (-2.0 * i / hd)
            a, b = v[h * hd + 2 * i], v[h * hd + 2 * i + 1]
            out[h * hd + 2 * i] = a * math.cos(th) - b * math.sin(th)
            out[h * hd + 2 * i + 1] = a * math.sin(th) + b * math.cos(th)
    return out


def _silu(z):
    return z / (1.0 + math.exp(-z))


def _block(cfg, W, pre, xs, pos, visible):
    """One pre-norm block over all rows xs at positions pos; row t attends to rows s with
    visible(t, s)."""
    H, hd, eps = cfg.n_heads, cfg.head_dim, cfg.rms_eps
    a = [_norm(x, W[pre + "attn_norm"], eps) for x in xs]
    q = [_rope(cfg, _matvec(W[pre + "wq"], a[t]), pos[t]) for t in range(len(xs))]
    k = [_rope(cfg, _matvec(W[pre + "wk"], a[t]), pos[t]) for t in range(len(xs))]
    v = [_matvec(W[pre + "wv"], a[t]) for t in range(len(xs))]
    out = []
    for t in range(len(xs)):
        o = [0.0] * (H * hd)
        keys = [s for s in range(len(xs)) if visible(t, s)]
        for h in range(H):
            sc = [sum(q[t][h * hd + j] * k[s][h * hd + j] for j in range(hd)) * cfg.attn_scale for s in keys]
            mx = max(sc)
            e = [math.exp(z - mx) for z in sc]
            tot = sum(e)
            for j in range(hd):
                o[h * hd + j] = sum(e[i] * v[s][h * hd + j] for i, s in enumerate(keys)) / tot
        hres = [xs[t][c] + val for c, val in enumerate(_matvec(W[pre + "wo"], o))]
        m = _norm(hres, W[pre + "mlp_norm"], eps)
        g1, g3 = _matvec(W[pre + "w1"], m), _matvec(W[pre + "w3"], m)
        mid = [_silu(g1[i]) * g3[i] for i in range(len(g1))]
        out.append([hres[c] + val for c, val in enumerate(_matvec(W[pre + "w2"], mid))])
    return out


def _stack(cfg, W, name, layers, xs, pos, visible):
    for l in range(layers):
        xs = _block(cfg, W, f"{name}.{l}.", xs, pos, visible)
    return xs


def _head(cfg, W, norm, y):
    return _matvec(W["unembed"], _norm(y, W[norm], cfg.rms_eps))


def _argmax(row):
    best = 0
    for i in range(1, len(row)):
        if row[i] > row[best]:
            best = i
    return best


def _prob(row, i):
    mx = max(row)
    return math.exp(row[i] - mx) / sum(math.exp(z - mx) for z in row)


def _bp_logit(W, h):
    hid = [_silu(sum(W["bp.w1"][j][c] * h[c] for c in range(len(h)))) for j in range(len(W["bp.w2"]))]
    return sum(W["bp.w2"][j] * hid[j] for j in range(len(hid))) + W["bp.bias"][0]


def brute_forward(cfg, W, x):
    """Every intermediate of the definition over bytes x."""
    T = len(x)
    causal = lambda t, s: s <= t  # noqa: E731
    h_e = _stack(cfg, W, "enc", cfg.n_enc, [list(W["embed"][c]) for c in x], list(range(T)), causal)
    if cfg.boundary == "learned":
        bnd = [_bp_logit(W, h_e[p]) > 0.0 for p in range(T)]
    else:
        bnd = [c == SP for c in x]
    Kp, k = [], 0
    for p in range(T):
        k += bnd[p]
        Kp.append(k)
    # closed segment k (1-based): after the (k-1)-th boundary up to and including the k-th
    z, start = [], 0
    for p in range(T):
        if bnd[p]:
            seg = range(start, p + 1)
            z.append([sum(h_e[q][c] for q in seg) / len(seg) for c in range(cfg.d_model)])
            start = p + 1
    u = [list(W["lm.bos"])] + z
    o = _stack(cfg, W, "lm", cfg.n_lm, u, list(range(len(u))), causal)
    y = _stack(cfg, W, "nb", cfg.n_nb, [[o[Kp[p]][c] + h_e[p][c] for c in range(cfg.d_model)] for p in range(T)],
               list(range(T)), causal)
    logits = [_head(cfg, W, "nb.norm", y[p]) for p in range(T)]
    return {"h_e": h_e, "b": bnd, "Kp": Kp, "z": z, "u": u, "o": o, "y": y, "nb": logits}


def brute_draft(cfg, W, x, n, F=None):
    """Drafter logits [n-1][256] at committed length t = len(x)."""
    F = F or brute_forward(cfg, W, x)
    t = len(x)
    if cfg.mb_kind == "mlp":
        rows = []
        for j in range(n - 1):
            v = list(F["y"][t - 1])
            for l in range(cfg.n_mb):
                s = _matvec(W[f"mlp.{j}.{l}.w"], v)
                v = [v[c] + _silu(s[c]) for c in range(len(v))]
            rows.append(_head(cfg, W, "mb.norm", v))
        return rows
    g_last = F["Kp"][t - 1]
    win = [q for q in range(t) if F["Kp"][q] >= g_last - 1]
    pos = win + list(range(t, t + n - 2))
    grp = [F["Kp"][q] for q in win] + [g_last] * (n - 2)
    rows = [[F["o"][g][c] + F["u"][g][c] for c in range(cfg.d_model)] for g in grp]
    vis = lambda i, j: j <= i and grp[j] in (grp[i], grp[i] - 1)  # noqa: E731
    h = _stack(cfg, W, "mb", cfg.n_mb, rows, pos, vis)
    return [_head(cfg, W, "mb.norm", r) for r in h[len(h) - (n - 1):]]


def brute_generate(cfg, W, prompt, n, tau, mode, G, force_cand=None):
    """The decode loop by full recompute. Returns (bytes, [accepted drafts per step]).
    force_cand(step): n bytes that replace the candidates of that step (the drafter still runs,
    and THRESH still tests its probabilities), to drive boundaries through the loop."""
    x = list(prompt)
    out, accepted = [], []
    step = 0
    while len(out) < G:
        F = brute_forward(cfg, W, x)
        c1 = _argmax(F["nb"][len(x) - 1])
        drafts, probs = [], []
        for row in brute_draft(cfg, W, x, n, F):
            drafts.append(_argmax(row))
            probs.append(_prob(row, drafts[-1]))
        cand = [c1] + drafts
        if force_cand is not None:
            cand = list(force_cand(step))
        step += 1
        a = 0
        if mode == THRESH:
            while a < n - 1 and probs[a] >= tau:
                a += 1
        else:
            nbv = brute_forward(cfg, W, x + cand)["nb"]
            while a < n - 1 and cand[1 + a] == _argmax(nbv[len(x) + a]):
                a += 1
        e = min(1 + a, G - len(out))
        x += cand[:e]
        out += cand[:e]
        accepted.append(a)
    return bytes(out), accepted


# ----------------------------------------------------------------------------- the pins
TEXT = b"ab cde f gh ijk l mn op"  # several closed segments, an open one, a one-byte word


@pytest.fixture(scope="module")
def lca():
    W = make_weights(CFG, 5)
    return W, as_model(CFG, W)


def test_forward_equals_scalar_chain(lca):
    W, M = lca
    B = brute_forward(CFG, W, TEXT)
    F = forward_full(M, TEXT)
    np.testing.assert_array_equal(F.Kp, B["Kp"])
    np.testing.assert_allclose(F.h_e, B["h_e"], rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(F.z, B["z"], rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(F.o, B["o"], rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(F.y, B["y"], rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(F.nb_logits, B["nb"], rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("t", [1, 2, 3, 6, 8, 12, 23])
def test_window_draft_equals_scalar_definition(lca, t):
    """t = 3 and 8 end on a boundary (the window spans the closed group and the boundary byte);
    t = 1, 2 lie in group 0 (no previous group)."""
    W, M = lca
    x = TEXT[:t]
    F = forward_full(M, x)
    got = mb_draft_logits(M, F.Kp, F.o, F.u, t, 4, x)
    want = brute_draft(CFG, W, x, 4)
    np.testing.assert_allclose(got, want, rtol=1e-9, atol=1e-9)


def test_mlp_heads_equal_scalar_definition():
    W = make_weights(CFG_MLP, 6)
    M = as_model(CFG_MLP, W)
    x = TEXT[:14]
    F = forward_full(M, x)
    got = mb_draft_logits(M, F.Kp, F.o, F.u, len(x), 4, x, y_last=F.y[-1])
    np.testing.assert_allclose(got, brute_draft(CFG_MLP, W, x, 4), rtol=1e-9, atol=1e-9)


def _tau_between(W, prompt, n):
    """A threshold that the first drafts of this prompt straddle (so that the loop both accepts
    and rejects)."""
    probs = sorted(_prob(r, _argmax(r)) for r in brute_draft(CFG, W, list(prompt), n))
    return 0.5 * (probs[0] + probs[-1])


@pytest.mark.parametrize("n", [2, 3, 5])
def test_thresh_generation_equals_scalar_loop(lca, n):
    W, M = lca
    prompt = TEXT[:10]
    G = 16
    tau = _tau_between(W, prompt, n) if n > 2 else 0.0
    want, acc = brute_generate(CFG, W, prompt, n, tau, THRESH, G)
    got, recs = generate_reference(M, prompt, n, tau, THRESH, G)
    assert got == want
    assert [r.a for r in recs] == acc
    dec = IncrementalDecoder(M)
    dec.prefill(prompt)
    inc = bytearray()
    while len(inc) < G:
        inc += dec.step(n, tau, THRESH, budget=G - len(inc)).emitted
    assert bytes(inc) == want
    if n == 2:
        assert all(a == 1 for a in acc[:-1])  # tau = 0 accepts every draft
    else:
        assert 0 < sum(acc) < (n - 1) * len(acc)  # the loop both accepts and rejects


def test_spec_generation_equals_scalar_loop(lca):
    W, M = lca
    prompt = TEXT[:9]
    want, acc = brute_generate(CFG, W, prompt, 3, 0.0, SPEC, 10)
    got, recs = generate_reference(M, prompt, 3, 0.0, SPEC, 10)
    assert got == want
    assert [r.a for r in recs] == acc


PATTERNS = [b"a b", b" c ", b"de ", b"  f", b"g h", b"ij "]


@pytest.mark.parametrize("mode", [THRESH, SPEC])
def test_loop_through_boundaries_equals_scalar_loop(lca, mode):
    """Candidates with spaces at every position (the greedy text of this random model holds none):
    segments close on accepted and on rejected bytes, so the LM module runs on latents that are
    then rolled back, and the window moves across groups. The cached decoder must keep exactly the
    accepted prefix of every cache."""
    from oracle import generate_incremental
    W, M = lca
    prompt = TEXT[:7]
    n, G = 3, 18
    tau = _tau_between(W, prompt, n)
    fc = lambda step: PATTERNS[step % len(PATTERNS)]  # noqa: E731
    want, acc = brute_generate(CFG, W, prompt, n, tau, mode, G, force_cand=fc)
    got, recs = generate_reference(M, prompt, n, tau, mode, G, force_cand=fc)
    assert got == want
    assert [r.a for r in recs] == acc
    inc, irecs = generate_incremental(M, prompt, n, tau, mode, G, force_cand=fc)
    assert inc == want
    assert [r.a for r in irecs] == acc
    assert want.count(SP) >= 3
    if mode == THRESH:
        assert 0 < sum(acc) < (n - 1) * len(acc)


# ----------------------------------------------------------------------------- learned boundaries
@pytest.fixture(scope="module")
def learned():
    """The learned predictor with its bias set so that about a third of the positions of the text
    end a segment (the scalar logits' upper tercile)."""
    W = make_weights(CFG_BP, 9)
    h = brute_forward(CFG, W, TEXT)["h_e"]
    lg = sorted(_bp_logit(W, r) for r in h)
    W["bp.bias"] = [-0.5 * (lg[2 * len(lg) // 3] + lg[2 * len(lg) // 3 - 1])]
    return W, as_model(CFG_BP, W)


def test_learned_boundaries_forward_equals_scalar_chain(learned):
    W, M = learned
    B = brute_forward(CFG_BP, W, TEXT)
    F = forward_full(M, TEXT)
    assert 4 <= sum(B["b"]) <= 12 and B["b"] != [c == SP for c in TEXT]
    np.testing.assert_array_equal(F.b, B["b"])
    np.testing.assert_array_equal(F.Kp, B["Kp"])
    np.testing.assert_allclose(F.z, B["z"], rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(F.o, B["o"], rtol=1e-10, atol=1e-10)
    np.testing.assert_allclose(F.nb_logits, B["nb"], rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("t", [1, 5, 9, 14, 23])
def test_learned_boundaries_window_equals_scalar_definition(learned, t):
    W, M = learned
    x = TEXT[:t]
    F = forward_full(M, x)
    got = mb_draft_logits(M, F.Kp, F.o, F.u, t, 4, x)
    np.testing.assert_allclose(got, brute_draft(CFG_BP, W, x, 4), rtol=1e-9, atol=1e-9)


@pytest.mark.parametrize("mode", [THRESH, SPEC])
def test_learned_boundaries_generation_equals_scalar_loop(learned, mode):
    """Segments close wherever the predictor fires on the encoder state of a candidate, accepted or
    rejected, so the LM module runs on speculative latents and the cached decoder rolls them back."""
    from oracle import generate_incremental
    W, M = learned
    prompt = TEXT[:8]
    n, G = 4, 16
    tau = 0.0
    if mode == THRESH:
        probs = sorted(_prob(r, _argmax(r)) for r in brute_draft(CFG_BP, W, list(prompt), n))
        tau = 0.5 * (probs[0] + probs[-1])
    want, acc = brute_generate(CFG_BP, W, prompt, n, tau, mode, G)
    got, recs = generate_reference(M, prompt, n, tau, mode, G)
    assert got == want
    assert [r.a for r in recs] == acc
    inc, irecs = generate_incremental(M, prompt, n, tau, mode, G)
    assert inc == want
    assert [r.a for r in irecs] == acc
    assert [(r.t, r.K) for r in irecs] == [(r.t, r.K) for r in recs]
    assert recs[-1].K > forward_full(M, prompt).Kp[-1]  # segments closed during generation
