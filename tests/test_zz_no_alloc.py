"""The allocation-free decode entry point (for callers that cannot allocate
device memory while they decode) against the regular one.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.  It also passes on its own in
a fresh process."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2607_28069_gb300.workloads import custom_spec, generate
from tests.helpers import attn_close, f64, oracle_layout, request_inputs, theta_of

SCRATCH_BYTES = 8 << 20   # the size of the library's built-in scratch array

pytestmark = pytest.mark.gpu


def _prepared_path():
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    spec = custom_spec(name="noalloc", layers=1, q_heads=28, kv_heads=4, head_dim=128,
                       rope_base=1e6, batch=3, pool_docs=5, docs_per_request=4,
                       doc_len=(300, 900), prefix_len=(10, 60), query_len=24, decode_steps=1)
    wl = generate(spec, device="cuda", gen_device="cpu")
    path = CacheHitPath(wl, with_lse=True)
    path.ttft_pass()
    return wl, path


def test_noalloc_decode_matches_workspace_decode_twice(cuda_lib):
    import paper_2607_28069_gb300 as pic
    wl, path = _prepared_path()
    # reference: the entry point with a caller workspace
    path.decode(0, 0)
    torch.cuda.synchronize()
    ref_out = f64(path.dec_out[0])
    ref_lse = f64(path.dec_lse[0])
    # two calls in a row through the allocation-free entry point (the second
    # sees the scratch the first one left behind)
    for call in range(2):
        out = torch.full_like(path.dec_out[0], float("nan"))
        lse = torch.full_like(path.dec_lse[0], float("nan"))
        pic.pic_attend_decode_noalloc(
            path.geom, 0, wl.q_dec[0, 0], wl.k_dec[0, 0], wl.v_dec[0, 0], path.ctx_len,
            wl.block_table, wl.num_pages, path.k_cache, path.v_cache, out, path.max_ctx,
            lse=lse, pos_offset=0)
        torch.cuda.synchronize()
        ok, max_abs, row = attn_close(f64(out), ref_out)
        assert ok, f"call {call}: err/bound {max_abs:.2f} row-rel {row:.2e}"
        assert np.abs(f64(lse) - ref_lse).max() < 5e-2
        # and against the oracle's decoding step over the same stitched context
        theta = theta_of(wl.spec)
        for b in range(wl.spec.batch):
            lay = oracle_layout(wl, b)
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, 0)
            K, V = O.dense_context(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), k, v,
                                   theta)
            (o_ref, lse_ref), _, _ = O.decode_step(
                K, V, f64(wl.q_dec[0, 0, b]), f64(wl.k_dec[0, 0, b]), f64(wl.v_dec[0, 0, b]),
                lay.ctx_len, theta, return_lse=True)
            ok, max_abs, row = attn_close(f64(out[b]), o_ref)
            assert ok, f"call {call} req {b}: err/bound {max_abs:.2f} row-rel {row:.2e}"
            assert np.abs(f64(lse[b]) - lse_ref).max() < 5e-2
    assert pic.pic_device_status() == (0, 0)


def test_noalloc_lowers_the_automatic_split_count_to_fit(cuda_lib):
    """16 query heads over one kv head at batch 32 and a ~10k-position
    context: the automatic split plan needs more partial states than the
    built-in array holds, so the allocation-free call lowers the split
    count to the largest that fits, and then gives exactly what the
    workspace entry point gives with that split count."""
    import paper_2607_28069_gb300 as pic
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    spec = custom_spec(name="noalloc_g16", layers=1, q_heads=16, kv_heads=1, head_dim=128,
                       rope_base=5e5, batch=32, pool_docs=4, docs_per_request=4,
                       doc_len=(2500, 2500), prefix_len=(16, 16), query_len=8, decode_steps=1)
    wl = generate(spec, device="cuda", gen_device="cpu")
    path = CacheHitPath(wl, with_lse=True)
    path.ttft_pass()
    B, mc = spec.batch, path.max_ctx
    auto = pic.pic_decode_num_splits(path.geom, B, mc, 0)
    fits = [s for s in range(1, auto + 1)
            if pic.pic_decode_workspace_size(path.geom, B, mc, s) <= SCRATCH_BYTES]
    assert fits and max(fits) < auto, (auto, fits[-3:])
    lowered = max(fits)
    ref_out = torch.empty_like(path.dec_out[0])
    ref_lse = torch.empty_like(path.dec_lse[0])
    ws = torch.empty(pic.pic_decode_workspace_size(path.geom, B, mc, lowered), dtype=torch.uint8,
                     device="cuda")
    pic.pic_attend_decode(path.geom, 0, wl.q_dec[0, 0], wl.k_dec[0, 0], wl.v_dec[0, 0],
                          path.ctx_len, wl.block_table, wl.num_pages, path.k_cache, path.v_cache,
                          ref_out, mc, ref_lse, lowered, ws, pos_offset=0)
    out = torch.full_like(ref_out, float("nan"))
    lse = torch.full_like(ref_lse, float("nan"))
    pic.pic_attend_decode_noalloc(path.geom, 0, wl.q_dec[0, 0], wl.k_dec[0, 0], wl.v_dec[0, 0],
                                  path.ctx_len, wl.block_table, wl.num_pages, path.k_cache,
                                  path.v_cache, out, mc, lse=lse, pos_offset=0)
    torch.cuda.synchronize()
    assert pic.pic_device_status() == (0, 0)
    assert torch.equal(out, ref_out) and torch.equal(lse, ref_lse)


def test_noalloc_rejects_scratch_beyond_its_array(cuda_lib):
    import paper_2607_28069_gb300 as pic
    wl, path = _prepared_path()
    out = torch.empty_like(path.dec_out[0])
    # 64 explicit splits over a 2^20-position bound needs far more than 8 MiB of partials
    big_batch = 600
    pos = torch.zeros(big_batch, dtype=torch.int32, device="cuda")
    bt = torch.zeros((big_batch, 1), dtype=torch.int32, device="cuda")
    q = torch.zeros((big_batch, 28, 128), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((big_batch, 4, 128), dtype=torch.bfloat16, device="cuda")
    o = torch.zeros((big_batch, 28, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(pic.PicError) as ei:
        pic.pic_attend_decode_noalloc(path.geom, 0, q, kv, kv, pos, bt, wl.num_pages,
                                      path.k_cache, path.v_cache, o, 1 << 20, num_splits=64)
    assert ei.value.status == 4 and "8388608" in str(ei.value)
    del out
