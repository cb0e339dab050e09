"""CPU oracle, part 1: the hierarchical byte LM with the LCA multi-byte head, in fp64.

TEST INFRASTRUCTURE ONLY. Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its ``cpu_baseline`` leg and ``--impl reference`` arm) may import
this package. The CUDA product path never calls it and shares no code with it;
both sides receive their inputs from ``synth`` alone.

Plain numpy float64, written for reading, not for speed. The model is the one of
Section 2.2 (encoder module, boundaries by the space rule or by a learned predictor
on the encoder states, mean-pool downsampling, LM module with a [BOS] latent,
upsampling by duplication, next-byte decoder) plus
the multi-byte head of Section 3 (LCA mask, residual r_2 added before
upsampling, shared unembedding). Blocks follow Llama 3 (Section 4.2): pre-norm
RMSNorm (eps 1e-6), rotary embeddings (base 1e5), SwiGLU MLP, no biases.

Readings taken where the paper is silent (each is also listed with the design notes):
  * K(p) counts boundaries at positions <= p, so a boundary byte receives the
    latent of the segment it closes (Algorithm 1 runs the LM module before the
    next-byte layers in the same iteration).
  * group g = the bytes with K(p) = g; the MB input of every byte of group g is
    o_g + u_g (u_0 = [BOS], u_k = z_k).
  * RoPE rotates interleaved pairs (2i, 2i+1) by pos * base^(-2i/h_d); byte
    modules use the byte position, the LM module the latent index.
  * no final norm on h_e or on the LM output; separate final RMSNorms for the
    next-byte and multi-byte heads; unembedding untied from the embedding.
  * argmax breaks ties toward the lowest byte value.
  * the learned boundary predictor is w_2 . SiLU(W_1 h_e[p]) + c, a boundary where its
    probability sigmoid(.) exceeds 0.5 (where the logit is positive).
"""
from __future__ import annotations

import numpy as np

from synth.configs import ModelConfig


# ----------------------------------------------------------------------------- block math
def rmsnorm(x, g, eps):
    """RMSNorm (Section 4.2): x / sqrt(mean(x^2) + eps) * g, over the last axis."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def silu(x):
    """SiLU(x) = x * sigmoid(x), the gate of the Llama-3 SwiGLU MLP."""
    with np.errstate(over="ignore"):
        return x / (1.0 + np.exp(-x))


def rope(x, pos, base):
    """Rotary embedding (Section 4.2, base 1e5): the pair (x[2i], x[2i+1]) of every
    head is rotated by the angle pos * base^(-2i/h_d). x: [T, H, h_d]; pos: [T]."""
    hd = x.shape[-1]
    inv = base ** (-np.arange(0, hd, 2, dtype=np.float64) / hd)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x0 = x[..., 0::2]
    x1 = x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def attend(q, k, v, mask, scale):
    """Softmax attention. q [T,H,h_d], k/v [S,H,h_d], mask [T,S] (True = key visible).
    One head at a time: scores q_h k_h^T * scale, masked softmax over keys, times v_h."""
    out = np.empty_like(q)
    for h in range(q.shape[1]):
        s = (q[:, h, :] @ k[:, h, :].T) * scale
        s = np.where(mask, s, -np.inf)
        s = s - s.max(axis=-1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=-1, keepdims=True)
        out[:, h, :] = p @ v[:, h, :]
    return out


def causal_mask(n_prev, n_new):
    """New row i (of n_new) sees all n_prev earlier rows and new rows <= i."""
    m = np.zeros((n_new, n_prev + n_new), dtype=bool)
    m[:, :n_prev] = True
    m[:, n_prev:] = np.tril(np.ones((n_new, n_new), dtype=bool))
    return m


def lca_mask(groups):
    """Latent Causal Attention mask (Section 3, Figure 2): query p sees key q iff
    q <= p and q lies in the same latent group as p or in the one just before it."""
    g = np.asarray(groups)
    T = len(g)
    q_le_p = np.tril(np.ones((T, T), dtype=bool))
    same_or_prev = (g[None, :] == g[:, None]) | (g[None, :] == g[:, None] - 1)
    return q_le_p & same_or_prev


def block(cfg: ModelConfig, lw, x, pos, mask, k_prev=None, v_prev=None):
    """One pre-norm Llama block over new rows x [T,d] at positions pos.
    k_prev/v_prev: post-RoPE keys/values [S0,H,h_d] of earlier rows (a KV cache);
    mask [T, S0+T]. Returns (x_out, k_new, v_new)."""
    T = x.shape[0]
    H, hd = cfg.n_heads, cfg.head_dim
    a = rmsnorm(x, lw["attn_norm"], cfg.rms_eps)
    q = rope((a @ lw["wq"].T).reshape(T, H, hd), pos, cfg.rope_base)
    k = rope((a @ lw["wk"].T).reshape(T, H, hd), pos, cfg.rope_base)
    v = (a @ lw["wv"].T).reshape(T, H, hd)
    K = k if k_prev is None else np.concatenate([k_prev, k], axis=0)
    V = v if v_prev is None else np.concatenate([v_prev, v], axis=0)
    att = attend(q, K, V, mask, cfg.attn_scale).reshape(T, H * hd)
    h = x + att @ lw["wo"].T
    m = rmsnorm(h, lw["mlp_norm"], cfg.rms_eps)
    h = h + (silu(m @ lw["w1"].T) * (m @ lw["w3"].T)) @ lw["w2"].T
    return h, k, v


# ----------------------------------------------------------------------------- model
class Model:
    """Weights as fp64 arrays plus the forward pieces of Section 2.2 and Section 3."""

    def __init__(self, cfg: ModelConfig, weights: dict):
        self.cfg = cfg
        self.w = {k: np.asarray(v, dtype=np.float64) for k, v in weights.items()}

    def layer(self, prefix, l):
        return {t: self.w[f"{prefix}.{l}.{t}"] for t in
                ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w1", "w3", "w2")}

    def n_layers(self, prefix):
        c = self.cfg
        return {"enc": c.n_enc, "lm": c.n_lm, "nb": c.n_nb, "mb": c.n_mb}[prefix]

    def run_stack(self, prefix, x, pos, mask_fn, caches=None):
        """Run all blocks of a stack. caches: list per layer of (k_prev, v_prev) or None.
        mask_fn(n_prev) gives the mask. Returns (x, [(k_new, v_new)] per layer)."""
        new = []
        for l in range(self.n_layers(prefix)):
            kp, vp = (None, None) if caches is None else caches[l]
            n_prev = 0 if kp is None else kp.shape[0]
            x, k, v = block(self.cfg, self.layer(prefix, l), x, pos, mask_fn(n_prev), kp, vp)
            new.append((k, v))
        return x, new

    def head(self, y, norm):
        """Final RMSNorm of a decoder head, then the shared unembedding (Section 3)."""
        return rmsnorm(y, self.w[norm], self.cfg.rms_eps) @ self.w["unembed"].T

    def embed(self, x):
        return self.w["embed"][np.frombuffer(bytes(x), dtype=np.uint8)]


def boundaries(cfg: ModelConfig, x):
    """Space rule: b_p = [x_p == 0x20]; the boundary byte is the last byte of its
    segment (used in place of the learned predictor of Section 2.2)."""
    return np.frombuffer(bytes(x), dtype=np.uint8) == cfg.boundary_byte


def boundary_logits(model: "Model", h):
    """Learned boundary predictor of Section 2.2 on encoder states h [T, d]: the logit of the
    boundary probability, w_2 . SiLU(W_1 h_p) + c."""
    w = model.w
    return silu(h @ w["bp.w1"].T) @ w["bp.w2"] + w["bp.bias"][0]


def boundary_flags(model: "Model", x, h_e):
    """b_p for bytes x with encoder states h_e (Algorithm 1, boundary step): the space rule on
    the bytes, or the learned predictor, b_p = [sigmoid(logit_p) > 0.5] = [logit_p > 0]."""
    if model.cfg.boundary == "learned":
        return boundary_logits(model, h_e) > 0.0
    return boundaries(model.cfg, x)


def latent_index_of(b):
    """K(p) = number of boundaries at positions <= p, from the flags b."""
    return np.cumsum(np.asarray(b, dtype=bool)).astype(np.int64)


def segments_of(b):
    """[(start, end)] inclusive byte ranges of the closed segments S_1..S_K (Section 2.2): each
    ends at a boundary and starts after the previous one."""
    segs, start = [], 0
    for p, f in enumerate(b):
        if f:
            segs.append((start, p))
            start = p + 1
    return segs


def latent_index(cfg: ModelConfig, x):
    """K(p) under the space rule."""
    return latent_index_of(boundaries(cfg, x))


def closed_segments(cfg: ModelConfig, x):
    """Closed segments under the space rule."""
    return segments_of(boundaries(cfg, x))


def group_start(cfg: ModelConfig, x, g):
    """First byte of group g: position 0 for g = 0, else the g-th boundary byte."""
    if g == 0:
        return 0
    return closed_segments(cfg, x)[g - 1][1]


def pool(h_e, segs):
    """Downsample by mean pooling over each closed segment, boundary byte included."""
    if not segs:
        return np.zeros((0, h_e.shape[1]))
    return np.stack([h_e[s:e + 1].mean(axis=0) for s, e in segs])


def window_draft_inputs(cfg: ModelConfig, Kp, o, u, t, n, x):
    """Rows of the MB window of Algorithm 1 (drafting step) at committed length t:
    the previous and the current group (from the first byte of group K(t-1)-1, or
    of group 0) then n-2 copies of the last row at positions t..t+n-3.
    The groups come from K(p) (x, the committed bytes, is not needed: group g >= 1 starts at
    its boundary byte, the first p with K(p) = g).
    Returns (inputs [W,d], positions [W], groups [W])."""
    g = int(Kp[t - 1])
    s = next(p for p in range(t) if Kp[p] >= g - 1) if g >= 1 else 0
    pos = list(range(s, t)) + list(range(t, t + n - 2))
    grp = [int(Kp[p]) for p in range(s, t)] + [g] * (n - 2)
    m = np.stack([o[k] + u[k] for k in grp])
    return m, np.asarray(pos), np.asarray(grp)


def mb_draft_logits(model: Model, Kp, o, u, t, n, x, y_last=None):
    """Logits [n-1, V] of the n-1 drafted bytes d_2..d_n (predicting x_{t+1}..x_{t+n-1}).
    LCA head (Section 3, Algorithm 1 drafting step): MB blocks over the window with the
    LCA mask, final RMSNorm, shared unembedding; only the last n-1 rows are kept.
    MLP head (Section 4.1, MLP-MBP): head j maps the last next-byte hidden state y_last
    through residual SiLU layers, then the MB norm and the unembedding."""
    cfg = model.cfg
    if n < 2:
        return np.zeros((0, cfg.vocab))
    if cfg.mb_kind == "mlp":
        rows = []
        for j in range(n - 1):
            v = y_last.copy()
            for l in range(cfg.n_mb):
                v = v + silu(model.w[f"mlp.{j}.{l}.w"] @ v)
            rows.append(v)
        return model.head(np.stack(rows), "mb.norm")
    m, pos, grp = window_draft_inputs(cfg, Kp, o, u, t, n, x)
    mask = lca_mask(grp)
    h, _ = model.run_stack("mb", m, pos, lambda n_prev: mask)
    return model.head(h[-(n - 1):], "mb.norm")


def full_sequence_lca_logits(model: Model, Kp, o, u, extra=0):
    """Training-style MB forward: every byte position p uses input o_{K(p)} + u_{K(p)}
    and the LCA mask over the whole sequence; ``extra`` rows duplicate the last group
    at the next positions. Row p predicts x_{p+2} (Eq. 2, shift-by-two target)."""
    grp = [int(k) for k in Kp] + [int(Kp[-1])] * extra
    m = np.stack([o[k] + u[k] for k in grp])
    pos = np.arange(len(grp))
    mask = lca_mask(grp)
    h, _ = model.run_stack("mb", m, pos, lambda n_prev: mask)
    return model.head(h, "mb.norm")


class Forward:
    """All intermediate values of one full forward over committed bytes x_0..x_{T-1}."""
    __slots__ = ("x", "h_e", "b", "Kp", "segs", "z", "u", "o", "y", "nb_logits", "caches")


def forward_full(model: Model, x, keep_caches=False):
    """Definition of the forward over bytes x (Section 2.2 and the forward part of Algorithm 1):
    embed, encoder (causal, RoPE at byte position) -> h_e; boundaries (space rule, or the
    learned predictor on h_e); mean-pool closed segments -> z_1..z_K; LM module over [BOS, z_1..z_K] (causal, RoPE at latent
    index) -> o_0..o_K; next-byte decoder over o_{K(p)} + h_e[p] (causal) -> y; final
    norm and unembedding -> next-byte logits (row p predicts x_{p+1})."""
    cfg = model.cfg
    T = len(x)
    F = Forward()
    F.x = bytes(x)
    pos = np.arange(T)
    causal = lambda n_prev: causal_mask(n_prev, T)
    F.h_e, enc_kv = model.run_stack("enc", model.embed(x), pos, causal)
    F.b = boundary_flags(model, x, F.h_e)
    F.Kp = latent_index_of(F.b)
    F.segs = segments_of(F.b)
    F.z = pool(F.h_e, F.segs)
    F.u = np.concatenate([model.w["lm.bos"][None, :], F.z], axis=0)
    K1 = F.u.shape[0]
    F.o, lm_kv = model.run_stack("lm", F.u, np.arange(K1), lambda n_prev: causal_mask(n_prev, K1))
    F.y, nb_kv = model.run_stack("nb", F.o[F.Kp] + F.h_e, pos, causal)
    F.nb_logits = model.head(F.y, "nb.norm")
    F.caches = {"enc": enc_kv, "lm": lm_kv, "nb": nb_kv} if keep_caches else None
    return F


def greedy(logits):
    """Lowest index among equal maxima."""
    return int(np.argmax(logits))


def max_prob(logits, idx):
    """softmax(logits)[idx] = exp(l_idx - logsumexp(l))."""
    mx = logits.max()
    return float(np.exp(logits[idx] - mx) / np.exp(logits - mx).sum())
