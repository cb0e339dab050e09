"""Paged KV caches on the GPU: every cache layer is a pool of 64-slot pages behind a per-sequence
page table, mapped at prefill for the prompts and by the decode steps as positions, latents and
multi-byte windows reach new pages. Results must not depend on where the pages lie: the decode
steps match the oracle across page boundaries, pools sized to exactly the pages a run maps give
bit-identical results to the default pools, and a pool one page short fails the step that needs
the page with LCA_E_CAPACITY and nothing else."""
import numpy as np
import pytest

from oracle import THRESH, IncrementalDecoder, Model
from synth import TINY, cached_weights, make_weights, words_text, zipf_text

pytestmark = pytest.mark.gpu

F32_TOL = 1e-4
BF16_TOL = 2e-2
SMALL_BF16 = TINY.replace(d_model=256, n_heads=4, head_dim=64, d_ff=1024, n_enc=1, n_lm=2,
                          n_nb=1, n_mb=2, dtype="bf16")


@pytest.fixture(scope="module")
def lca():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2608_15454_gb300 import build, lca as mod
    build.build()
    mod.load_library()
    return mod


def check_tables(ctx, decs):
    """Page-table invariants: every committed position, latent and window row of a sequence is
    mapped; no page is mapped twice; the pool's counter equals the pages mapped."""
    seen = set()
    for cache in range(3):
        tab, used, pages = ctx.page_table(cache)
        mapped = tab[tab >= 0]
        assert len(set(mapped.tolist())) == mapped.size, cache
        assert mapped.size == used <= pages
        assert mapped.max(initial=-1) < pages
        seen.add((cache, used))
        for b, d in enumerate(decs):
            if cache == 0:
                need = d.t
            elif cache == 1:
                need = d.K + 1
            else:
                continue  # window rows: checked through the logits
            assert (tab[b, :(need + 63) // 64] >= 0).all(), (cache, b, need)
    return seen


def test_ragged_batch_across_page_boundaries_tiny_fp32(lca):
    """fp32 storage, four sequences whose positions (62, 127, 1 and 63 bytes of prompt) and
    latents (31 spaces in the last prompt, three more per step) cross 64-slot page boundaries
    during the run, so later pages interleave between sequences: bytes, accepted counts, t, K
    and group starts bit-exact, logits within 1e-4."""
    W = cached_weights(TINY)
    prompts = [words_text(0, 62), words_text(1, 127), b"a", b"a " * 31 + b"a"]
    n = 3
    ctx = lca.Context(TINY, W, max_batch=4, max_bytes=400, max_n=n)
    ctx.prefill(prompts)
    decs = []
    for p in prompts:
        d = IncrementalDecoder(Model(TINY, W))
        d.prefill(p)
        decs.append(d)
    for s in range(24):
        cands = [bytes([97 + (s + b) % 26, 32 if (s + b) % 2 else 98, 99]) for b in range(3)] + [b"   "]
        a = [s % 3, 2, (s + 1) % 3, 2]
        ctx.force_candidates(cands, n)
        ctx.force_accept(a)
        recs = [d.step(n, 0.75, THRESH, forced=a[b], forced_cand=cands[b]) for b, d in enumerate(decs)]
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        for b, (d, r) in enumerate(zip(decs, recs)):
            np.testing.assert_allclose(nb[b], r.nb_logits, atol=F32_TOL, rtol=0)
            np.testing.assert_allclose(mb[b], r.mb_logits, atol=F32_TOL, rtol=0)
            assert out[b] == r.emitted
            st = ctx.state(b)
            assert (st["t"], st["K"]) == (d.t, d.K)
            assert (st["prev_group_start"], st["group_start"]) == d.group_starts()
    assert decs[0].t > 64 and decs[1].t > 128 and decs[3].K + 1 > 64
    check_tables(ctx, decs)
    # the decode steps mapped pages in step order: sequence 0's second page does not follow its first
    tab, _, _ = ctx.page_table(0)
    assert tab[0, 1] != tab[0, 0] + 1
    ctx.close()


def _steps(lca, ctx, steps, n, batch):
    """Forced candidates and accepted counts; the logs of the steps up to the first failing one,
    and its status (None: every step returned LCA_OK)."""
    logs = []
    for s in range(steps):
        cands = [bytes([97 + (s + b) % 26, 32 if (s + b) % 2 == 0 else 98, 99, 32]) for b in range(batch)]
        ctx.force_candidates(cands, n)
        ctx.force_accept([(s + b) % n for b in range(batch)])
        try:
            out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        except lca.LcaError as e:
            return logs, e.status
        nb, mb = ctx.logits(n)
        logs.append((out, nb.copy(), mb.copy()))
    return logs, None


def _run(lca, model, W, prompts, steps, n, **pools):
    ctx = lca.Context(model, W, max_batch=len(prompts), max_bytes=900, max_n=n, **pools)
    ctx.prefill(prompts)
    logs, status = _steps(lca, ctx, steps, n, len(prompts))
    assert status is None
    return ctx, logs


def test_exact_pools_bit_identical_and_exhaustion(lca):
    """bf16 storage at d = 256, three sequences: pools of exactly the pages a run maps reproduce
    the default pools' bytes and logits bit for bit; with one byte-cache page fewer, the step that
    needs it returns LCA_E_CAPACITY, and a new prefill starts from empty pools again."""
    W = make_weights(SMALL_BF16, gain=8.0, seed=5)
    prompts = [zipf_text(0, 300), zipf_text(1, 60) + b" ", zipf_text(2, 129)]
    n, steps = 4, 16
    ctx, ref = _run(lca, SMALL_BF16, W, prompts, steps, n)
    used = [ctx.page_table(c)[1] for c in range(3)]
    ctx.close()
    ctx, got = _run(lca, SMALL_BF16, W, prompts, steps, n, kv_pages=used[0], lm_pages=used[1],
                    mb_pages=used[2])
    for (o1, nb1, mb1), (o2, nb2, mb2) in zip(ref, got):
        assert o1 == o2
        assert np.array_equal(nb1, nb2) and np.array_equal(mb1, mb2)
    assert [ctx.page_table(c)[1] for c in range(3)] == used
    ctx.close()
    # one byte page short: the prompts fit, a later step does not
    prompt_pages = sum((len(p) + 63) // 64 for p in prompts)
    assert used[0] - 1 >= prompt_pages
    ctx = lca.Context(SMALL_BF16, W, max_batch=3, max_bytes=900, max_n=n, kv_pages=used[0] - 1,
                      lm_pages=used[1], mb_pages=used[2])
    ctx.prefill(prompts)
    logs, failed = _steps(lca, ctx, steps, n, len(prompts))
    assert failed == lca.LCA_E_CAPACITY
    # the steps before the one that needed the missing page are the default pools' steps
    assert 0 < len(logs) < steps
    for (o1, nb1, mb1), (o2, nb2, mb2) in zip(ref, logs):
        assert o1 == o2 and np.array_equal(nb1, nb2) and np.array_equal(mb1, mb2)
    short = [prompts[0][:100], prompts[1], prompts[2]]
    ctx.prefill(short)
    assert ctx.page_table(0)[1] == sum((len(p) + 63) // 64 for p in short)
    ctx.step(n, 0.75, lca.LCA_THRESH)
    ctx.close()
    # prompts that do not fit the pool: the prefill refuses them
    ctx = lca.Context(SMALL_BF16, W, max_batch=3, max_bytes=900, max_n=n, kv_pages=prompt_pages - 1)
    with pytest.raises(lca.LcaError) as e:
        ctx.prefill(prompts)
    assert e.value.status == lca.LCA_E_CAPACITY
    ctx.close()


def test_batch32_tensor_core_attention_over_interleaved_pages(lca):
    """32 sequences x 4 heads: the tensor-core attention kernels (prefill tiles and the decode
    kernel over tensor maps of the page pools) read pages that the decode steps map in between
    other sequences' pages. Logits within the bf16 tolerance of the oracle, bytes and state equal."""
    W = make_weights(SMALL_BF16, gain=8.0, seed=7)
    rng = np.random.default_rng(3)
    lens = rng.integers(40, 200, size=32)
    prompts = [zipf_text(10 + b, int(L)) for b, L in enumerate(lens)]
    n = 4
    ctx = lca.Context(SMALL_BF16, W, max_batch=32, max_bytes=400, max_n=n)
    ctx.prefill(prompts)
    decs = []
    for p in prompts:
        d = IncrementalDecoder(Model(SMALL_BF16, W))
        d.prefill(p)
        decs.append(d)
    for s in range(8):
        cands = [bytes([97 + (s + b) % 26, 32 if (s + b) % 3 == 0 else 98, 99, 100]) for b in range(32)]
        a = [(s + b) % n for b in range(32)]
        ctx.force_candidates(cands, n)
        ctx.force_accept(a)
        recs = [d.step(n, 0.75, THRESH, forced=a[b], forced_cand=cands[b]) for b, d in enumerate(decs)]
        out, cnt = ctx.step(n, 0.75, lca.LCA_THRESH)
        nb, mb = ctx.logits(n)
        for b, (d, r) in enumerate(zip(decs, recs)):
            np.testing.assert_allclose(nb[b], r.nb_logits, atol=BF16_TOL * 8, rtol=0)
            np.testing.assert_allclose(mb[b], r.mb_logits, atol=BF16_TOL * 8, rtol=0)
            assert out[b] == r.emitted
            st = ctx.state(b)
            assert (st["t"], st["K"]) == (d.t, d.K)
    check_tables(ctx, decs)
    ctx.close()
