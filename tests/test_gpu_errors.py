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


def test_bounded_wait_that_runs_out_returns_timeout(lca):
    """The first weight wait of the weight-streaming GEMV is cut to zero spins, so it reports late
    at once (its second wait, with the full budget, still drains the copies): the step returns
    LCA_E_TIMEOUT without a hang or a fault. With the hook cleared, a new prefill gives the same
    bytes as a context that never timed out."""
    from synth import make_weights, zipf_text
    model = TINY.replace(d_model=256, n_heads=4, head_dim=64, d_ff=1024, n_enc=1, n_lm=2, n_nb=1, n_mb=2,
                         dtype="bf16")
    W = make_weights(model, gain=8.0, seed=5)
    p = zipf_text(0, 300)
    lib = lca.load_library()
    ref = lca.Context(model, W, max_batch=1, max_bytes=400, max_n=4)
    ref.prefill([p])
    want = [ref.step(3, 0.75) for _ in range(3)]
    ref.close()
    ctx = lca.Context(model, W, max_batch=1, max_bytes=400, max_n=4)
    ctx.prefill([p])
    assert lib.lca_debug_set_wait_spins(0) == 0
    try:
        with pytest.raises(lca.LcaError) as e:
            ctx.step(3, 0.75)
        assert e.value.status == -7
    finally:
        assert lib.lca_debug_set_wait_spins(-1) == 0
    ctx.prefill([p])
    got = [ctx.step(3, 0.75) for _ in range(3)]
    for (o1, c1), (o2, c2) in zip(got, want):
        assert o1 == o2 and list(c1) == list(c2)
    ctx.close()
