"""Brute-force pin of the oracle's block (CPU): one pre-norm Llama block (Section 4.2) written as
scalar loops over explicit indices, from the definitions, on tiny random inputs:

  a = x / sqrt(mean(x^2) + eps) * g_attn
  q_t[h*hd + j] = sum_c Wq[h*hd + j][c] a_t[c]   (likewise k, v); head h owns features h*hd .. h*hd+hd-1
  RoPE: features (2i, 2i+1) of a head rotate by pos * base^(-2i/hd)
  o_t[h*hd + j] = sum_{s visible to t} softmax_s(q_t . k_s * scale) v_s[h*hd + j]
  h_t = x_t + Wo o_t
  y_t = h_t + W2 (silu(W1 m_t) * (W3 m_t)),  m = RMSNorm(h_t) * g_mlp

and compared with the oracle's vectorised block, with and without a key/value cache."""
import math
import random

import numpy as np

from oracle.model import block
from synth.configs import ModelConfig

CFG = ModelConfig(d_model=8, n_heads=2, head_dim=4, d_ff=12, n_enc=1, n_lm=1, n_nb=1, n_mb=1,
                  dtype="f32")


def _rand(rng, *shape, scale=0.5):
    return np.array([rng.gauss(0.0, scale) for _ in range(int(np.prod(shape)))]).reshape(shape)


def _weights(rng):
    d, f = CFG.d_model, CFG.d_ff
    return {"attn_norm": 1.0 + _rand(rng, d, scale=0.2), "wq": _rand(rng, d, d), "wk": _rand(rng, d, d),
            "wv": _rand(rng, d, d), "wo": _rand(rng, d, d), "mlp_norm": 1.0 + _rand(rng, d, scale=0.2),
            "w1": _rand(rng, f, d), "w3": _rand(rng, f, d), "w2": _rand(rng, d, f)}


def _norm(v, g, eps):
    ms = sum(e * e for e in v) / len(v)
    r = 1.0 / math.sqrt(ms + eps)
    return [v[c] * r * g[c] for c in range(len(v))]


def _matvec(W, v):
    return [sum(W[o][c] * v[c] for c in range(len(v))) for o in range(len(W))]


def _rope(v, pos):
    out = list(v)
    H, hd = CFG.n_heads, CFG.head_dim
    for h in range(H):
        for i in range(hd // 2):
            th = pos * CFG.rope_base ** (-2.0 * i / hd)
            a, b = v[h * hd + 2 * i], v[h * hd + 2 * i + 1]
            out[h * hd + 2 * i] = a * math.cos(th) - b * math.sin(th)
            out[h * hd + 2 * i + 1] = a * math.sin(th) + b * math.cos(th)
    return out


def _brute_block(W, xs, pos, visible):
    """xs: rows; pos: their positions; visible(t, s): row t sees key row s (over all rows)."""
    H, hd, eps = CFG.n_heads, CFG.head_dim, CFG.rms_eps
    wl = {k: W[k].tolist() for k in W}
    a = [_norm(x, wl["attn_norm"], eps) for x in xs]
    q = [_rope(_matvec(wl["wq"], a[t]), pos[t]) for t in range(len(xs))]
    k = [_rope(_matvec(wl["wk"], a[t]), pos[t]) for t in range(len(xs))]
    v = [_matvec(wl["wv"], a[t]) for t in range(len(xs))]
    out = []
    for t in range(len(xs)):
        o = [0.0] * (H * hd)
        for h in range(H):
            keys = [s for s in range(len(xs)) if visible(t, s)]
            sc = [sum(q[t][h * hd + j] * k[s][h * hd + j] for j in range(hd)) * CFG.attn_scale for s in keys]
            mx = max(sc)
            e = [math.exp(z - mx) for z in sc]
            tot = sum(e)
            for j in range(hd):
                o[h * hd + j] = sum(e[i] * v[s][h * hd + j] for i, s in enumerate(keys)) / tot
        hres = [xs[t][c] + val for c, val in enumerate(_matvec(wl["wo"], o))]
        m = _norm(hres, wl["mlp_norm"], eps)
        g1, g3 = _matvec(wl["w1"], m), _matvec(wl["w3"], m)
        mid = [g1[i] / (1.0 + math.exp(-g1[i])) * g3[i] for i in range(len(g1))]
        out.append([hres[c] + val for c, val in enumerate(_matvec(wl["w2"], mid))])
    return out


def test_block_equals_scalar_definition_causal():
    rng = random.Random(11)
    W = _weights(rng)
    T = 5
    x = _rand(rng, T, CFG.d_model, scale=1.0)
    pos = [3, 4, 5, 6, 7]
    mask = np.tril(np.ones((T, T), dtype=bool))
    got, _, _ = block(CFG, W, x, np.array(pos), mask)
    want = _brute_block(W, x.tolist(), pos, lambda t, s: s <= t)
    np.testing.assert_allclose(got, np.array(want), rtol=1e-12, atol=1e-12)


def test_block_with_cache_equals_scalar_definition_over_all_rows():
    """Rows 0..2 first, then rows 3..5 against their cached keys and values: the new rows equal the
    scalar block over all six rows (a cache changes nothing), here with a non-causal visibility
    pattern (row 4 skips key 1) to pin the mask orientation."""
    rng = random.Random(12)
    W = _weights(rng)
    x = _rand(rng, 6, CFG.d_model, scale=1.0)
    pos = [0, 1, 2, 3, 4, 5]

    def visible(t, s):
        return s <= t and not (t == 4 and s == 1)

    full = np.array([[visible(t, s) for s in range(6)] for t in range(6)])
    _, k0, v0 = block(CFG, W, x[:3], np.array(pos[:3]), full[:3, :3])
    got, _, _ = block(CFG, W, x[3:], np.array(pos[3:]), full[3:, :], k0, v0)
    want = _brute_block(W, x.tolist(), pos, visible)[3:]
    np.testing.assert_allclose(got, np.array(want), rtol=1e-12, atol=1e-12)
