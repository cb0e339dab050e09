"""lca_decode_attention_noalloc: the decode attention for callers that cannot allocate device
memory (plugin hosts that pass only input and output buffers, code that must not call an
allocator). Its scratch is a fixed array inside the library; these tests check, through the C
ABI, that two calls in a row give the same output as lca_decode_attention with caller scratch, for
both cache types and both head sizes, and that an out-of-range cache length is reported by the
status call of either form.

This file is collected last on purpose, so that a run stopping at the first failure has run
every other test before it.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _setup():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_15454_gb300 import build, lca
    build.build()
    lca.load_library()
    return torch, lca


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("hd", [32, 64])
def test_noalloc_attention_matches_scratch_version_twice(dtype, hd):
    torch, lca = _setup()
    B, H, S, n_rows, splits = 2, 1024 // hd, 700, 5, 8
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    g = torch.Generator(device="cuda").manual_seed(11 + hd)
    scale = 1.0 / hd ** 0.5
    scratch = torch.empty(lca.decode_attention_scratch_bytes(B, H, hd, splits), dtype=torch.uint8,
                          device="cuda")
    assert lca.decode_attention_scratch_bytes(B, H, hd, splits) <= lca.load_library() \
        .lca_decode_attention_noalloc_capacity()
    for call in range(2):
        q = torch.randn(B * n_rows, H * hd, device="cuda", generator=g)
        k = torch.randn(B, H, S, hd, device="cuda", generator=g).to(tdt)
        v = torch.randn(B, H, S, hd, device="cuda", generator=g).to(tdt)
        lens = torch.randint(1, S + 1, (B * n_rows,), device="cuda", generator=g, dtype=torch.int32)
        want = torch.empty_like(q)
        got = torch.full_like(q, float("nan"))
        assert lca.decode_attention(q, want, k, v, lens, scale, splits, scratch) == 0
        assert lca.decode_attention_status(scratch) == 0
        assert lca.decode_attention(q, got, k, v, lens, scale, splits, noalloc=True) == 0
        assert lca.decode_attention_status(noalloc=True) == 0
        torch.cuda.synchronize()
        np.testing.assert_allclose(got.cpu().numpy(), want.cpu().numpy(), atol=1e-4, rtol=0)


def test_out_of_range_cache_length_is_reported_by_both_forms():
    """A kv_len beyond the cache reads only the cache's slots and is reported as
    LCA_E_DEVICE_STATE by the status call; the next good call clears it."""
    torch, lca = _setup()
    B, H, hd, S, n_rows, splits = 1, 16, 64, 96, 3, 4
    g = torch.Generator(device="cuda").manual_seed(5)
    q = torch.randn(B * n_rows, H * hd, device="cuda", generator=g)
    k = torch.randn(B, H, S, hd, device="cuda", generator=g).to(torch.bfloat16)
    v = torch.randn(B, H, S, hd, device="cuda", generator=g).to(torch.bfloat16)
    bad = torch.tensor([S, S + 7, 10], device="cuda", dtype=torch.int32)
    good = torch.tensor([S, S, 10], device="cuda", dtype=torch.int32)
    scratch = torch.empty(lca.decode_attention_scratch_bytes(B, H, hd, splits), dtype=torch.uint8, device="cuda")
    ref, o1, o2 = torch.empty_like(q), torch.empty_like(q), torch.empty_like(q)
    assert lca.decode_attention(q, ref, k, v, good, 0.125, splits, scratch) == 0
    assert lca.decode_attention_status(scratch) == 0
    assert lca.decode_attention(q, o1, k, v, bad, 0.125, splits, scratch) == 0
    assert lca.decode_attention_status(scratch) == -5
    assert lca.decode_attention(q, o2, k, v, bad, 0.125, splits, noalloc=True) == 0
    assert lca.decode_attention_status(noalloc=True) == -5
    np.testing.assert_allclose(o1.cpu().numpy(), ref.cpu().numpy(), atol=1e-5, rtol=0)
    np.testing.assert_allclose(o2.cpu().numpy(), ref.cpu().numpy(), atol=1e-5, rtol=0)
    assert lca.decode_attention(q, o2, k, v, good, 0.125, splits, noalloc=True) == 0
    assert lca.decode_attention_status(noalloc=True) == 0


def test_noalloc_attention_rejects_sizes_beyond_its_array():
    torch, lca = _setup()
    lib = lca.load_library()
    B, H, hd, S = 64, 16, 64, 8
    q = torch.zeros(B, H * hd, device="cuda")
    k = torch.zeros(B, H, S, hd, device="cuda", dtype=torch.bfloat16)
    lens = torch.ones(B, device="cuda", dtype=torch.int32)
    assert lca.decode_attention_scratch_bytes(B, H, hd, 16) > lib.lca_decode_attention_noalloc_capacity()
    out = torch.empty_like(q)
    assert lca.decode_attention(q, out, k, k, lens, 0.125, 16, noalloc=True) == -2
