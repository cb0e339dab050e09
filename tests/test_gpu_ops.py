"""The decode-attention kernel as a standalone call against a plain PyTorch fp32 reference."""
import numpy as np
import pytest

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


def reference(q, k, v, kv_len, scale, n_rows):
    """fp32 softmax attention: row r of sequence b over cache slots [0, kv_len[r])."""
    import torch
    B, H, S, hd = k.shape
    out = torch.zeros_like(q)
    kf, vf = k.float(), v.float()
    for r in range(q.shape[0]):
        b, L = r // n_rows, int(kv_len[r])
        qr = q[r].view(H, hd)
        s = torch.einsum("hd,hsd->hs", qr, kf[b, :, :L]) * scale
        p = torch.softmax(s, dim=-1)
        out[r] = torch.einsum("hs,hsd->hd", p, vf[b, :, :L]).reshape(-1)
    return out


def make_case(dtype, B, H, hd, S, n_rows, seed):
    import torch
    g = torch.Generator(device="cuda").manual_seed(seed)
    q = torch.randn(B * n_rows, H * hd, device="cuda", generator=g)
    k = torch.randn(B, H, S, hd, device="cuda", generator=g).to(dtype)
    v = torch.randn(B, H, S, hd, device="cuda", generator=g).to(dtype)
    lens = torch.randint(1, S + 1, (B * n_rows,), device="cuda", generator=g, dtype=torch.int32)
    lens[0] = S            # full cache
    lens[-1] = 1           # one key
    return q, k, v, lens


@pytest.mark.parametrize("dtype_name,hd,splits,n_rows", [("float32", 32, 1, 3), ("bfloat16", 64, 8, 7),
                                                         ("bfloat16", 64, 16, 20), ("float32", 64, 3, 1)])
def test_decode_attention_matches_fp32_reference(lca, dtype_name, hd, splits, n_rows):
    import torch
    dtype = getattr(torch, dtype_name)
    B, H, S = 3, 4, 301
    q, k, v, lens = make_case(dtype, B, H, hd, S, n_rows, seed=hd + splits)
    out = torch.empty_like(q)
    nbytes = lca.decode_attention_scratch_bytes(B, H, hd, splits)
    scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    scale = 1.0 / hd ** 0.5
    assert lca.decode_attention(q, out, k, v, lens, scale, splits, scratch) == 0
    torch.cuda.synchronize()
    want = reference(q, k, v, lens, scale, n_rows)
    np.testing.assert_allclose(out.cpu().numpy(), want.cpu().numpy(), atol=1e-4, rtol=0)


def test_decode_attention_rejects_bad_arguments(lca):
    import torch
    q, k, v, lens = make_case(torch.float32, 1, 2, 32, 16, 2, seed=0)
    out = torch.empty_like(q)
    small = torch.empty(256, dtype=torch.uint8, device="cuda")
    assert lca.decode_attention(q, out, k, v, lens, 0.1, 4, small) == -2
    assert lca.decode_attention(q, out, k, v, lens, 0.1, 99, small) == -1


@pytest.mark.parametrize("M,Mused,N,K,typ", [
    (128, 128, 64, 64, 0),          # one tile, one K block
    (200, 200, 128, 1024, 0),       # 128-column tiles, split K in a cluster
    (300, 257, 1024, 1024, 0),      # ragged rows, cluster split K
    (64, 17, 192, 4096, 0),         # few rows, deep K
    (1024, 1000, 3072, 1024, 0),    # eight row tiles in TMEM at once
    (256, 200, 3072, 1024, 0),      # 128-column tiles, four-way split K
    (2100, 2050, 512, 1024, 128),   # launch shaped for 128 rows: clustered CTAs walk 17 row tiles
    (700, 650, 3072, 1024, 256),    # two row tiles per CTA, 256-column tiles
    (2100, 2100, 256, 320, 0),      # more row tiles than TMEM holds; K blocks not a power of two
    # skinny GEMM (weights as the MMA's M operand) for at most 64 typical rows
    (32, 32, 1024, 1024, 0),        # 16-way cluster split K, one K block per CTA
    (32, 19, 8192, 1024, 0),        # ragged rows, two-way split K
    (64, 50, 3072, 1024, 0),        # 64-row tiles, four-way split K
    (300, 257, 1024, 4096, 32),     # launch shaped for 32 rows: clusters walk nine row tiles
    (200, 200, 256, 1088, 64),      # 17 K blocks (no split), ring wraps, ragged last row tile
    (48, 48, 2048, 2048, 48),       # partial 64-row tile
])
def test_tensor_core_gemm_matches_reference(lca, M, Mused, N, K, typ):
    """tcgen05 GEMMs (TMA weight tiles, 128-byte swizzle, TMEM accumulators, split bf16
    activations, cluster split-K; activations as the M operand, or the weights for few rows)
    against a float64 product of the fp32 activations and the bf16 weights."""
    import torch
    g = torch.Generator(device="cuda").manual_seed(M + N + K)
    x = torch.randn(M, K, device="cuda", generator=g)
    W = (torch.randn(N, K, device="cuda", generator=g) * 0.05).to(torch.bfloat16)
    y = torch.full((M, N), float("nan"), device="cuda")
    Md = torch.tensor([Mused], dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    scratch = torch.empty(lca.debug_gemm_scratch_bytes(M, K), dtype=torch.uint8, device="cuda")
    assert lca.debug_gemm(x, W, y, Md, err, rows_typ=typ, scratch=scratch) == 0
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    want = (x[:Mused].double() @ W.double().t()).cpu().numpy()
    got = y[:Mused].double().cpu().numpy()
    # two bf16 halves keep ~2^-17 of each activation; fp32 accumulation over K terms
    tol = 1e-5 * float(np.abs(want).max())
    np.testing.assert_allclose(got, want, atol=tol, rtol=0)
    assert torch.isnan(y[Mused:]).all()
