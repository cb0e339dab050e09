"""Model shapes and workloads of the multi-byte-prediction (MBP) decode step.

This module only names sizes. It holds none of the method's arithmetic and is
shared, together with the seeded generators in ``synth.data``, by the CPU oracle
and the CUDA path.

Model shape: the hierarchical byte LM of Section 2.2 (encoder, LM module,
next-byte decoder) with the multi-byte head of Section 3, layer split of the
hyper-parameter table (Appendix A: LCA-MBP 2/16/2/2, MLP-MBP 2/16/2/3), hidden
size 1024 and inner size 4096 (Section 4.2), RMSNorm eps 1e-6 and RoPE base 1e5
(Section 4.2). The head count is 16 x 64 (the paper states 8 heads; the
workloads below fix 16 x 64).
"""
from __future__ import annotations

import dataclasses
import json
import os
from dataclasses import dataclass, field

BOUNDARY_BYTE = 0x20
VOCAB = 256


@dataclass(frozen=True)
class ModelConfig:
    d_model: int
    n_heads: int
    head_dim: int
    d_ff: int
    n_enc: int
    n_lm: int
    n_nb: int
    n_mb: int            # LCA head: transformer blocks; MLP head: residual layers per head
    mb_kind: str = "lca"  # "lca" | "mlp"
    n_mlp_heads: int = 0  # MLP head only: independent heads (drafts per step = heads)
    dtype: str = "f32"    # "f32" | "bf16": storage type of weights and KV caches
    boundary: str = "space"  # "space": byte rule | "learned": predictor on the encoder states
    d_bp: int = 0         # learned predictor only: hidden width of its MLP
    boundary_byte: int = BOUNDARY_BYTE
    rope_base: float = 1.0e5
    rms_eps: float = 1.0e-6
    vocab: int = VOCAB

    @property
    def attn_scale(self) -> float:
        return 1.0 / (self.head_dim ** 0.5)

    def replace(self, **kw) -> "ModelConfig":
        return dataclasses.replace(self, **kw)


@dataclass(frozen=True)
class Workload:
    name: str
    model: ModelConfig
    batch: int
    prompt_len: int
    gen: int
    n_list: tuple
    tau_list: tuple
    text: str                 # "words" (uniform letters) | "zipf" (5k-word lexicon)
    oracle_seqs: tuple = (0,)  # sequences the CPU oracle replays at full size
    gain_key: str = ""        # key into gains.json (unembedding gain for ~50% acceptance)

    @property
    def max_n(self) -> int:
        return max(self.n_list)

    @property
    def max_bytes(self) -> int:
        return self.prompt_len + self.gen + self.max_n


TINY = ModelConfig(d_model=128, n_heads=4, head_dim=32, d_ff=512,
                   n_enc=1, n_lm=2, n_nb=1, n_mb=1, dtype="f32")

PAPER = ModelConfig(d_model=1024, n_heads=16, head_dim=64, d_ff=4096,
                    n_enc=2, n_lm=16, n_nb=2, n_mb=2, dtype="bf16")

PAPER_MLP = PAPER.replace(mb_kind="mlp", n_mb=3, n_mlp_heads=6)

# The external verifier of Section 6.3 (FxT): a learned boundary predictor (hidden width d), a
# four-layer next-byte decoder and no multi-byte head.
FXT = PAPER.replace(boundary="learned", d_bp=1024, n_nb=4, n_mb=0)

WORKLOADS = {
    "tiny_b1": Workload("tiny_b1", TINY, batch=1, prompt_len=256, gen=128,
                        n_list=(3,), tau_list=(0.75,), text="words",
                        oracle_seqs=(0,), gain_key="tiny"),
    "paper_b1": Workload("paper_b1", PAPER, batch=1, prompt_len=1024, gen=512,
                         n_list=(3, 4, 5, 6, 7), tau_list=(0.75,), text="zipf",
                         oracle_seqs=(0,), gain_key="paper"),
    "paper_b32": Workload("paper_b32", PAPER, batch=32, prompt_len=2048, gen=512,
                          n_list=(4,), tau_list=(0.75,), text="zipf",
                          oracle_seqs=(0, 1), gain_key="paper"),
    "paper_long_b8": Workload("paper_long_b8", PAPER, batch=8, prompt_len=8192, gen=256,
                              n_list=(5,), tau_list=(0.5, 0.75, 0.9), text="zipf",
                              oracle_seqs=(0,), gain_key="paper"),
    "mlp_b128": Workload("mlp_b128", PAPER_MLP, batch=128, prompt_len=1024, gen=256,
                         n_list=(7,), tau_list=(0.75,), text="zipf",
                         oracle_seqs=(0, 1, 2, 3), gain_key="paper_mlp"),
}

_GAINS_PATH = os.path.join(os.path.dirname(__file__), "gains.json")


def load_gains() -> dict:
    """Unembedding gains chosen on the oracle: g (W_u <- g * W_u) so that about half of the
    drafted bytes pass tau = 0.75, and s (the boundary byte's row of W_u times s) so that
    generated text holds spaces at the prompts' rate. Written by ``oracle/calibrate_gain.py``."""
    if not os.path.exists(_GAINS_PATH):
        return {}
    with open(_GAINS_PATH) as f:
        return json.load(f)


def gain_for(workload: Workload, calibrated: bool) -> float:
    return weight_gains(workload, calibrated)["gain"]


def weight_gains(workload: Workload, calibrated: bool) -> dict:
    """Keyword arguments of make_weights for a workload: {"gain": g, "space_gain": s}, both 1
    for the literal random-init weights."""
    if not calibrated:
        return {"gain": 1.0, "space_gain": 1.0}
    g = load_gains().get(workload.gain_key)
    if g is None:
        raise KeyError(f"no calibrated gain for {workload.gain_key!r}; run oracle/calibrate_gain.py")
    if not isinstance(g, dict):
        return {"gain": float(g), "space_gain": 1.0}
    return {"gain": float(g["gain"]), "space_gain": float(g.get("space_gain", 1.0))}
