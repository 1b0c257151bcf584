"""The allocation-free decode entry point (for callers that cannot allocate
device memory while they decode) against the regular one.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.  It also passes on its own in
a fresh process."""
import numpy as np
import pytest
import torch

from paper_2607_28069_gb300.workloads import custom_spec, generate
from tests.helpers import attn_close, f64

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
        assert ok, f"call {call}: max-abs {max_abs:.2e} row-rel {row:.2e}"
        assert np.abs(f64(lse) - ref_lse).max() < 5e-2
    assert pic.pic_device_status() == (0, 0)


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
