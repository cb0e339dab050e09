"""Seeded synthetic inputs: byte prompts and random-init weights.

Shared by the CPU oracle and the CUDA path. Holds no arithmetic of the method:
only random draws, a fixed tensor order, and bf16 rounding of the drawn values
(so that both sides receive identical numbers for the bf16 model).

Text stands in for the paper's evaluation prompts (CNN/DailyMail, CoQA, IFEval,
Opus-100; Section 4.3), which are not used:
  * "words": lowercase words of uniform length 1..10, letters uniform a..z,
    joined by single spaces;
  * "zipf":  words drawn with probability proportional to rank^-1.1 from a
    lexicon of 5,000 distinct random lowercase words of length 1..12, joined by
    single spaces (mean patch about 8.5 bytes, space included: the Zipf-weighted
    mean word length of this lexicon plus one).
Weights: standard normal x 0.02 drawn in a fixed tensor order from
numpy.random.default_rng(0); RMSNorm gains are 1.
"""
from __future__ import annotations

import functools

import numpy as np

from .configs import ModelConfig, Workload

INIT_STD = 0.02
_LEXICON_SIZE = 5000
_ZIPF_S = 1.1


# ----------------------------------------------------------------------------- text
def words_text(seq: int, length: int) -> bytes:
    rng = np.random.default_rng(1000 + seq)
    out = bytearray()
    while len(out) < length:
        n = int(rng.integers(1, 11))
        w = (rng.integers(0, 26, size=n) + ord("a")).astype(np.uint8).tobytes()
        if out:
            out += b" "
        out += w
    return bytes(out[:length])


@functools.lru_cache(maxsize=1)
def lexicon() -> tuple:
    rng = np.random.default_rng(7)
    words, seen = [], set()
    while len(words) < _LEXICON_SIZE:
        n = int(rng.integers(1, 13))
        w = (rng.integers(0, 26, size=n) + ord("a")).astype(np.uint8).tobytes()
        if w not in seen:
            seen.add(w)
            words.append(w)
    return tuple(words)


@functools.lru_cache(maxsize=1)
def _zipf_probs() -> np.ndarray:
    r = np.arange(1, _LEXICON_SIZE + 1, dtype=np.float64)
    p = r ** (-_ZIPF_S)
    return p / p.sum()


def zipf_text(seq: int, length: int) -> bytes:
    lex = lexicon()
    p = _zipf_probs()
    rng = np.random.default_rng(1000 + seq)
    out = bytearray()
    while len(out) < length:
        for i in rng.choice(_LEXICON_SIZE, size=256, p=p):
            if out:
                out += b" "
            out += lex[int(i)]
            if len(out) >= length:
                break
    return bytes(out[:length])


def prompt(workload: Workload, seq: int, length: int | None = None) -> bytes:
    n = workload.prompt_len if length is None else length
    if workload.text == "words":
        return words_text(seq, n)
    if workload.text == "zipf":
        return zipf_text(seq, n)
    raise ValueError(workload.text)


def prompts(workload: Workload, seqs=None, length: int | None = None) -> list:
    seqs = range(workload.batch) if seqs is None else seqs
    return [prompt(workload, s, length) for s in seqs]


# ----------------------------------------------------------------------------- weights
BLOCK_TENSORS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w1", "w3", "w2")


def block_shapes(cfg: ModelConfig) -> dict:
    d, f = cfg.d_model, cfg.d_ff
    return {"attn_norm": (d,), "wq": (d, d), "wk": (d, d), "wv": (d, d), "wo": (d, d),
            "mlp_norm": (d,), "w1": (f, d), "w3": (f, d), "w2": (d, f)}


def tensor_list(cfg: ModelConfig) -> list:
    """(name, shape) in the fixed draw order. Linear weights are [out, in]."""
    d, v = cfg.d_model, cfg.vocab
    bs = block_shapes(cfg)
    out = [("embed", (v, d))]

    def stack(prefix, n):
        for l in range(n):
            for t in BLOCK_TENSORS:
                out.append((f"{prefix}.{l}.{t}", bs[t]))

    stack("enc", cfg.n_enc)
    out.append(("lm.bos", (d,)))
    stack("lm", cfg.n_lm)
    stack("nb", cfg.n_nb)
    out.append(("nb.norm", (d,)))
    if cfg.mb_kind == "lca":
        stack("mb", cfg.n_mb)
    elif cfg.mb_kind == "mlp":
        for j in range(cfg.n_mlp_heads):
            for l in range(cfg.n_mb):
                out.append((f"mlp.{j}.{l}.w", (d, d)))
    else:
        raise ValueError(cfg.mb_kind)
    out.append(("mb.norm", (d,)))
    out.append(("unembed", (v, d)))
    if cfg.boundary == "learned":  # drawn last, so the other tensors do not change
        out += [("bp.w1", (cfg.d_bp, d)), ("bp.w2", (cfg.d_bp,)), ("bp.bias", (1,))]
    return out


def is_norm(name: str) -> bool:
    return name.endswith("norm")


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), kept as float32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> 16) & 1) + np.uint32(0x7FFF)
    return ((u + bias) & np.uint32(0xFFFF0000)).view(np.float32)


def make_weights(cfg: ModelConfig, gain: float = 1.0, seed: int = 0, space_gain: float = 1.0,
                 bp_bias: float = 0.0) -> dict:
    """name -> float32 array. For dtype "bf16" every value is bf16-representable.
    ``gain`` multiplies the unembedding before rounding (acceptance calibration);
    ``space_gain`` multiplies its row of the boundary byte first (boundary-rate calibration);
    ``bp_bias`` is the learned boundary predictor's output bias (its boundary rate)."""
    rng = np.random.default_rng(seed)
    out = {}
    for name, shape in tensor_list(cfg):
        if is_norm(name):
            a = np.ones(shape, dtype=np.float32)
        elif name == "bp.bias":
            a = np.full(shape, bp_bias, dtype=np.float32)
        else:
            a = rng.standard_normal(shape, dtype=np.float32)
            a *= np.float32(INIT_STD)
        if name == "unembed" and space_gain != 1.0:
            a[cfg.boundary_byte] *= np.float32(space_gain)
        if name == "unembed" and gain != 1.0:
            a = (a * np.float32(gain)).astype(np.float32)
        if cfg.dtype == "bf16" and not is_norm(name):
            a = round_bf16(a)
        out[name] = a
    return out


@functools.lru_cache(maxsize=4)
def cached_weights(cfg: ModelConfig, gain: float = 1.0, seed: int = 0, space_gain: float = 1.0) -> dict:
    return make_weights(cfg, gain, seed, space_gain)


def param_count(cfg: ModelConfig) -> int:
    return int(sum(int(np.prod(s)) for _, s in tensor_list(cfg)))
