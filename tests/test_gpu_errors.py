"""Failure paths of the C ABI on a GPU, made on the host: arguments over capacity, calls out
of order, missing weights, and a non-finite weight planted in the host copy (the head flags
non-finite logits through the device error word; nothing faults or hangs)."""
import numpy as np
import pytest

from synth import TINY, cached_weights, words_text

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lca():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_15454_gb300 import build, lca as mod
    build.build()
    mod.load_library()
    return mod


def test_capacity_and_order(lca):
    W = cached_weights(TINY)
    ctx = lca.Context(TINY, W, max_batch=2, max_bytes=300, max_n=4)
    with pytest.raises(lca.LcaError) as e:
        ctx.step(3, 0.75)
    assert e.value.status == -8                      # step before prefill
    with pytest.raises(lca.LcaError) as e:
        ctx.prefill([words_text(0, 299)])            # prompt + max_n > max_bytes
    assert e.value.status == -2
    with pytest.raises(lca.LcaError) as e:
        ctx.prefill([b"a b", b"c", b"d"])            # batch > max_batch
    assert e.value.status == -2
    ctx.prefill([words_text(0, 100), b"x y"])
    with pytest.raises(lca.LcaError) as e:
        ctx.step(5, 0.75)                            # n > max_n
    assert e.value.status == -2
    out, cnt = ctx.step(4, 0.75)                     # still usable after the errors
    assert all(1 <= c <= 4 for c in cnt)
    ctx.close()


def test_missing_weight_is_rejected(lca):
    W = dict(cached_weights(TINY))
    W.pop("nb.norm")
    with pytest.raises(lca.LcaError) as e:
        lca.Context(TINY, W, max_batch=1, max_bytes=300, max_n=4)
    assert e.value.status == -3


def test_non_finite_weight_returns_numeric_error(lca):
    W = {k: np.array(v, copy=True) for k, v in cached_weights(TINY).items()}
    W["unembed"][7, 3] = np.nan
    ctx = lca.Context(TINY, W, max_batch=1, max_bytes=300, max_n=4)
    with pytest.raises(lca.LcaError) as e:
        ctx.prefill([words_text(0, 100)])
        ctx.step(3, 0.75)
    assert e.value.status == -6
    ctx.close()
