"""Model shapes against the numbers the paper prints (``tests/golden/``)."""
import os

from synth import PAPER, param_count
from synth.configs import FXT, PAPER_MLP

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _layer_table():
    rows = {}
    for line in open(os.path.join(GOLDEN, "paper_layer_table.txt")):
        if line.strip() and not line.startswith("#"):
            name, *v = line.split()
            rows[name] = tuple(int(x) for x in v)
    return rows


def _layers(cfg):
    return (cfg.n_enc, cfg.n_lm, cfg.n_nb, cfg.n_mb)


def test_layer_splits_are_the_papers():
    t = _layer_table()
    assert _layers(PAPER) == t["LCA-MBP"]
    assert _layers(PAPER_MLP) == t["MLP-MBP"]
    assert _layers(FXT) == t["FxT"] and FXT.boundary == "learned"
    assert len(t) == 5 and t["LlamaByte"] == (22, 0, 0, 0)


def test_verifier_is_about_the_drafters_size():
    """Section 6.3 verifies with a baseline of the same size: FxT's two extra next-byte layers
    replace the two multi-byte layers (the predictor adds d^2 + 2d)."""
    d = PAPER.d_model
    assert param_count(FXT) - param_count(PAPER) == d * d + d + 1
