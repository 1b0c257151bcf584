"""GPU parity: every step of the cache-hit path through the C ABI against the
CPU oracle on the same seeded inputs.

Bars (written here; derived from bf16 rounding and the fp32 arithmetic):
* layout, slot map, inline positions, ctx: bit-exact;
* V and every copied value: bit-exact;
* relocated / rotated K: |g - r| <= 4e-3 max(|r|, 2^-8 rowmax) and row rel-L2 <= 4e-3;
* attention outputs: |g - r| <= 1e-2 + half a bf16 ulp at max(|g|, |r|) and per-row
  rel-L2 <= 2e-2 against the exact fp64 oracle (peaked cases: against its
  bf16-storage mode).
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2607_28069_gb300.workloads import WORKLOADS, custom_spec, generate
from tests.helpers import (attn_close, f64, kv_tolerance_ok, oracle_layout, request_inputs,
                           theta_of, half_ulp_bf16)

pytestmark = pytest.mark.gpu

SMALL = {
    "tiny": WORKLOADS["tiny"],
    "llama8b_1layer": WORKLOADS["llama8b_1layer"],
    "ragged_b3": custom_spec(name="ragged_b3", layers=2, q_heads=8, kv_heads=2, head_dim=128,
                             rope_base=5e5, batch=3, pool_docs=6, docs_per_request=4,
                             doc_len=(1, 300), prefix_len=(0, 40), query_len=37),
    "gqa7_decode": custom_spec(name="gqa7_decode", layers=2, q_heads=28, kv_heads=4,
                               head_dim=128, rope_base=1e6, batch=2, pool_docs=4,
                               docs_per_request=3, doc_len=(100, 700), prefix_len=(5, 70),
                               query_len=20, decode_steps=3),
    "d64_g8": custom_spec(name="d64_g8", layers=1, q_heads=16, kv_heads=2, head_dim=64,
                          rope_base=1e4, batch=2, pool_docs=5, docs_per_request=5,
                          doc_len=(30, 200), prefix_len=(16, 16), query_len=64, decode_steps=2),
    "g16_decode": custom_spec(name="g16_decode", layers=1, q_heads=32, kv_heads=2,
                              head_dim=128, rope_base=5e5, batch=2, pool_docs=3,
                              docs_per_request=2, doc_len=(200, 400), prefix_len=(8, 8),
                              query_len=5, decode_steps=2),
    # prefix rows fill four of five query pairs: the split plan gives them one
    # CTA each and the rest to the pair that sees the documents
    "long_prefix": custom_spec(name="long_prefix", layers=1, q_heads=32, kv_heads=8,
                               head_dim=128, rope_base=5e5, batch=1, pool_docs=4,
                               docs_per_request=3, doc_len=(400, 600), prefix_len=(300, 300),
                               query_len=20, decode_steps=1),
    # post-document inline spans S_k (canonical order P, D_1, S_1, ..., D_m,
    # S_m, Q), some of them empty
    "spans_b2": custom_spec(name="spans_b2", layers=2, q_heads=8, kv_heads=2, head_dim=128,
                            rope_base=5e5, batch=2, pool_docs=5, docs_per_request=4,
                            doc_len=(20, 300), prefix_len=(0, 40), query_len=24,
                            span_len=(0, 3), decode_steps=2),
    "spans_d64": custom_spec(name="spans_d64", layers=1, q_heads=16, kv_heads=2, head_dim=64,
                             rope_base=1e4, batch=2, pool_docs=6, docs_per_request=6,
                             doc_len=(5, 130), prefix_len=(3, 17), query_len=9,
                             span_len=(0, 150), decode_steps=1),
    # boundary states around every document (header and trailer blocks of
    # a boundary-conditioned cache), supplied as pool entries 0 and 1 and
    # repeated in the request's order: H, D, T, H, D, T, ...
    "boundary_blocks": custom_spec(name="boundary_blocks", layers=1, q_heads=8, kv_heads=2,
                                   head_dim=128, rope_base=5e5, batch=2, pool_docs=5,
                                   docs_per_request=9, doc_len=(3, 90), prefix_len=(5, 20),
                                   query_len=12, fixed_order=(0, 2, 1, 0, 3, 1, 0, 4, 1),
                                   span_len=(0, 4), decode_steps=1),
    # 80 short documents per request: a long document table (the deviation
    # kernel keeps it in shared memory)
    "many_docs": custom_spec(name="many_docs", layers=1, q_heads=8, kv_heads=2, head_dim=128,
                             rope_base=5e5, batch=1, pool_docs=80, docs_per_request=80,
                             doc_len=(4, 40), prefix_len=(2, 8), query_len=16, decode_steps=1),
    "no_docs": custom_spec(name="no_docs", layers=1, q_heads=4, kv_heads=1, head_dim=64,
                           rope_base=1e4, batch=2, pool_docs=1, docs_per_request=0,
                           doc_len=(10, 10), prefix_len=(3, 30), query_len=9, decode_steps=1),
    # documents compiled at per-document base positions (Eq. 3 moves a key from
    # any base a to its target b): bases 0..2000 against targets up to ~1200,
    # so some documents move forwards and some backwards (delta < 0)
    "base_mixed": custom_spec(name="base_mixed", layers=2, q_heads=8, kv_heads=2, head_dim=128,
                              rope_base=5e5, batch=3, pool_docs=6, docs_per_request=4,
                              doc_len=(1, 300), prefix_len=(0, 40), query_len=29,
                              base_pos=(0, 2000), decode_steps=2),
    # bases beyond 1.2e5 behind short targets: delta ~ -1.3e5, the angle
    # range of the ~139k-token requests, with spans and d = 64
    "base_far_spans": custom_spec(name="base_far_spans", layers=1, q_heads=16, kv_heads=2,
                                  head_dim=64, rope_base=1e4, batch=2, pool_docs=5,
                                  docs_per_request=5, doc_len=(5, 200), prefix_len=(3, 17),
                                  query_len=9, span_len=(0, 40), base_pos=(120000, 140000),
                                  decode_steps=1),
    "base_far_d128": custom_spec(name="base_far_d128", layers=1, q_heads=32, kv_heads=8,
                                 head_dim=128, rope_base=5e5, batch=1, pool_docs=8,
                                 docs_per_request=8, doc_len=(100, 600), prefix_len=(64, 64),
                                 query_len=64, base_pos=(130000, 145000), decode_steps=1),
}

_CACHE = {}


def run_path(name, prefill_splits=0, decode_splits=0, rope_style=0):
    key = (name, prefill_splits, decode_splits, rope_style)
    if key in _CACHE:
        return _CACHE[key]
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    import paper_2607_28069_gb300 as pic
    wl = generate(SMALL[name], device="cuda", gen_device="cpu")
    path = CacheHitPath(wl, prefill_splits=prefill_splits, decode_splits=decode_splits,
                        with_lse=True, rope_style=rope_style)
    path.ttft_pass()
    dec = []
    if wl.q_dec is not None:
        for s in range(wl.spec.decode_steps):
            path.decode_pass(s)
            dec.append((path.dec_out.clone(), path.dec_lse.clone()))
    code, detail = pic.pic_device_status()
    assert code == 0, f"device status {code} detail {detail}"
    _CACHE[key] = (wl, path, dec)
    return _CACHE[key]


def _style(rope_style):
    return O.INTERLEAVED if rope_style else O.HALF


@pytest.mark.parametrize("name", list(SMALL))
def test_compose_bit_exact(cuda_lib, name):
    wl, path, _ = run_path(name)
    off, dl = path.doc_offset.cpu().numpy(), path.doc_delta.cpu().numpy()
    slots, ipos = path.slot_mapping.cpu().numpy(), path.inline_pos.cpu().numpy()
    ctx = path.ctx_len.cpu().numpy()
    for b in range(wl.spec.batch):
        lay = oracle_layout(wl, b)
        m = len(lay.doc_ids)
        assert ctx[b] == lay.ctx_len
        assert list(off[b, :m]) == lay.doc_offset
        assert list(dl[b, :m]) == lay.doc_delta
        assert (off[b, m:] == -1).all()
        assert np.array_equal(slots[b, :lay.ctx_len], lay.slot_mapping)
        assert (slots[b, lay.ctx_len:] == -1).all()
        tin = len(lay.inline_pos)
        assert np.array_equal(ipos[b, :tin], lay.inline_pos)
        assert (ipos[b, tin:] == -1).all()


@pytest.mark.parametrize("rope_style", [0, 1])
@pytest.mark.parametrize("name", ["tiny", "llama8b_1layer", "ragged_b3", "d64_g8", "spans_b2",
                                  "spans_d64", "boundary_blocks", "base_mixed", "base_far_spans",
                                  "base_far_d128"])
def test_stitched_cache(cuda_lib, name, rope_style):
    """Relocated doc keys within the K bar, values bit-exact, inline K rotated
    at their positions, inline V bit-exact -- all read back through the slots."""
    wl, path, _ = run_path(name, rope_style=rope_style)
    theta = theta_of(wl.spec)
    for layer in range(wl.spec.layers):
        for b in range(wl.spec.batch):
            lay = oracle_layout(wl, b)
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
            K, V = O.dense_context(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), k, v,
                                   theta, _style(rope_style))
            slots = torch.as_tensor(lay.slot_mapping, device="cuda")
            kc = path.k_cache[layer].reshape(-1, wl.spec.kv_heads, 16, wl.spec.head_dim)
            vc = path.v_cache[layer].reshape(-1, wl.spec.kv_heads, 16, wl.spec.head_dim)
            Kg = f64(kc[slots // 16, :, slots % 16])
            Vg = f64(vc[slots // 16, :, slots % 16])
            ok, ratio = kv_tolerance_ok(Kg, K)
            assert ok, f"K layer {layer} req {b}: worst err/bound {ratio:.3f}"
            assert np.array_equal(Vg, V), "V must be a bit copy"


@pytest.mark.parametrize("base", [0, 40])
def test_delta_zero_is_bit_exact(cuda_lib, base):
    """A document whose target equals its base (delta 0) keeps its keys bit
    for bit: compiled at 0 with no prefix, and at 40 behind a 40-token prefix."""
    spec = custom_spec(name="delta0", layers=1, q_heads=4, kv_heads=2, head_dim=128,
                       rope_base=5e5, batch=1, pool_docs=1, docs_per_request=1,
                       doc_len=(77, 77), prefix_len=(base, base), query_len=3,
                       base_pos=(base, base))
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(spec, device="cuda", gen_device="cpu")
    assert int(wl.doc_base_pos[0]) == base
    path = CacheHitPath(wl)
    path.compose()
    path.relocate()
    torch.cuda.synchronize()
    assert int(path.doc_delta[0, 0]) == 0 and int(path.doc_offset[0, 0]) == base
    slots = path.slot_mapping[0, base:base + 77]
    kc = path.k_cache[0].reshape(-1, 2, 16, 128)
    assert torch.equal(kc[slots // 16, :, slots % 16], wl.k_pool[0, :77])


@pytest.mark.parametrize("name", list(SMALL))
def test_prefill_attention(cuda_lib, name):
    wl, path, _ = run_path(name)
    theta = theta_of(wl.spec)
    for layer in range(wl.spec.layers):
        for b in range(wl.spec.batch):
            lay = oracle_layout(wl, b)
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
            (o_ref, lse_ref), _, _ = O.cache_hit_prefill(
                lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), q, k, v, theta,
                return_lse=True)
            tin = q.shape[0]
            o_gpu = f64(path.out[layer, b, :tin])
            ok, max_abs, row = attn_close(o_gpu, o_ref)
            assert ok, f"layer {layer} req {b}: err/bound {max_abs:.2f} row-rel {row:.2e}"
            lse_gpu = f64(path.lse[layer, b, :tin])
            assert np.abs(lse_gpu - lse_ref).max() < 5e-2


@pytest.mark.parametrize("splits", [1, 2, 5, 32])
def test_prefill_split_count_invariance(cuda_lib, splits):
    wl, path, _ = run_path("llama8b_1layer", prefill_splits=splits)
    wl0, path0, _ = run_path("llama8b_1layer")
    theta = theta_of(wl.spec)
    lay = oracle_layout(wl, 0)
    docs, k_docs, v_docs, q, k, v = request_inputs(wl, 0, 0)
    o_ref, _, _ = O.cache_hit_prefill(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(),
                                      q, k, v, theta)
    o_gpu = f64(path.out[0, 0, :q.shape[0]])
    ok, max_abs, row = attn_close(o_gpu, o_ref)
    assert ok, f"splits {splits}: err/bound {max_abs:.2f} row-rel {row:.2e}"
    # Split counts differ in rounding only: the outputs are bf16, so two
    # counts may round a value to neighbouring bf16 values (one spacing apart).
    a, b0 = f64(path.out), f64(path0.out)
    bar = np.maximum(1e-2, 2 * half_ulp_bf16(np.maximum(np.abs(a), np.abs(b0))))
    assert (np.abs(a - b0) <= bar).all(), np.abs(a - b0).max()


@pytest.mark.parametrize("name", ["gqa7_decode", "d64_g8", "g16_decode", "no_docs", "spans_b2",
                                  "base_mixed", "base_far_spans", "base_far_d128"])
@pytest.mark.parametrize("splits", [0, 1, 3])
def test_decode_steps(cuda_lib, name, splits):
    wl, path, dec = run_path(name, decode_splits=splits)
    theta = theta_of(wl.spec)
    for layer in range(wl.spec.layers):
        for b in range(wl.spec.batch):
            lay = oracle_layout(wl, b)
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
            K, V = O.dense_context(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), k, v, theta)
            for s, (out_s, lse_s) in enumerate(dec):
                (o_ref, lse_ref), K, V = O.decode_step(
                    K, V, f64(wl.q_dec[s, layer, b]), f64(wl.k_dec[s, layer, b]),
                    f64(wl.v_dec[s, layer, b]), lay.ctx_len + s, theta, return_lse=True)
                ok, max_abs, row = attn_close(f64(out_s[layer, b]), o_ref)
                assert ok, f"step {s} layer {layer} req {b}: {max_abs:.2e} {row:.2e}"
                assert np.abs(f64(lse_s[layer, b]) - lse_ref).max() < 5e-2


def test_decode_matches_prefill_last_row(cuda_lib):
    """A decode step over the cache equals the prefill row of the same token."""
    wl, path, dec = run_path("gqa7_decode", decode_splits=1)
    # Oracle-free property: redo step 0 as a one-token prefill of a fresh path.
    theta = theta_of(wl.spec)
    lay = oracle_layout(wl, 0)
    docs, k_docs, v_docs, q, k, v = request_inputs(wl, 0, 0)
    K, V = O.dense_context(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), k, v, theta)
    qd = f64(wl.q_dec[0, 0, 0])
    o_dec, K2, V2 = O.decode_step(K, V, qd, f64(wl.k_dec[0, 0, 0]), f64(wl.v_dec[0, 0, 0]),
                                  lay.ctx_len, theta)
    o_pre = O.attention(O.rotary(qd[None], lay.ctx_len, theta), np.array([lay.ctx_len]), K2, V2)
    np.testing.assert_allclose(o_dec, o_pre[0], atol=1e-12)
    ok, max_abs, row = attn_close(f64(dec[0][0][0, 0]), o_pre[0])
    assert ok, (max_abs, row)


def test_needle_and_peaked_softmax(cuda_lib):
    """Outputs of size O(1): a planted needle (found only if layout, re-rotation
    and attention are all right) and queries scaled x4 for a peaked softmax."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(WORKLOADS["llama8b_1layer"], device="cpu", gen_device="cpu")
    theta = theta_of(wl.spec)
    lay = oracle_layout(wl, 0)
    wl.q_inline.mul_(4.0)
    # needle: doc #3 of the request, token 100, aligned with query head 0 of the last token
    qpos = int(lay.inline_pos[-1])
    d3 = wl.meta["docs"][0][3]
    tgt = lay.doc_offset[3] + 100
    qrot = O.rotary(f64(wl.q_inline[0, 0, -1, 0]), qpos, theta)
    needle_t = 3.0 * qrot / np.linalg.norm(qrot) * np.sqrt(128)
    raw = O.rotary(needle_t, -tgt, theta)
    row = int(wl.doc_token_start[d3]) + 100
    wl.k_pool[0, row, 0] = torch.as_tensor(O.rotary(raw, 100, theta), dtype=torch.bfloat16)
    for name in ("doc_len", "doc_base_pos", "doc_token_start", "k_pool", "v_pool", "req_doc_ids",
                 "req_num_docs", "prefix_len", "query_len", "block_table", "q_inline",
                 "k_inline", "v_inline", "inline_len"):
        setattr(wl, name, getattr(wl, name).cuda())
    path = CacheHitPath(wl, with_lse=True)
    path.ttft_pass()
    docs, k_docs, v_docs, q, k, v = request_inputs(wl, 0, 0)
    # peaked scores: compare with the bf16-storage oracle (cache and queries in bf16)
    o_ref, _, _ = O.cache_hit_prefill(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(),
                                      q, k, v, theta, storage="bf16")
    o_gpu = f64(path.out[0, 0, :q.shape[0]])
    ok, max_abs, rowrel = attn_close(o_gpu, o_ref, abs_tol=1e-2, row_rel=1e-2)
    assert ok, (max_abs, rowrel)
    v_needle = f64(wl.v_pool[0, row, 0])
    assert np.linalg.norm(o_gpu[-1, 0] - v_needle) < 0.1 * np.linalg.norm(v_needle)


def test_device_checks_report_bad_inputs(cuda_lib):
    import paper_2607_28069_gb300 as pic
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(WORKLOADS["tiny"], device="cuda", gen_device="cpu")
    path = CacheHitPath(wl)
    wl.req_doc_ids[0, 1] = 7            # pool has 2 docs
    path.compose()
    code, detail = pic.pic_device_status()
    assert code == 1 and detail == 0 and int(path.ctx_len[0]) == -1
    wl.req_doc_ids[0, 1] = 1
    wl.block_table[0, 9] = -1           # page of positions 144..159 missing
    path.compose()
    code, _ = pic.pic_device_status()
    assert code == 6
    assert pic.pic_device_status() == (0, 0)   # cleared by the read


def test_decode_reports_a_context_beyond_max_ctx(cuda_lib):
    """max_ctx bounds the decode split plan: a token whose keys reach past it
    is a device-checked error (context overflow), not a silent truncation."""
    import paper_2607_28069_gb300 as pic
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL["g16_decode"], device="cuda", gen_device="cpu")
    path = CacheHitPath(wl, decode_splits=1)
    path.ttft_pass()
    torch.cuda.synchronize()
    assert pic.pic_device_status() == (0, 0)
    short = int(path.ctx_len.max()) + 1 - 16      # one page short of the new token
    ws = torch.empty(pic.pic_decode_workspace_size(path.geom, wl.spec.batch, short, 1),
                     dtype=torch.uint8, device="cuda")
    pic.pic_attend_decode(path.geom, 0, wl.q_dec[0, 0], wl.k_dec[0, 0], wl.v_dec[0, 0],
                          path.ctx_len, wl.block_table, wl.num_pages, path.k_cache, path.v_cache,
                          path.dec_out[0], short, None, 1, ws)
    code, _ = pic.pic_device_status()
    assert code == 4
    # the same call with a sufficient bound is clean
    path.decode(0, 0)
    assert pic.pic_device_status() == (0, 0)


# ------------------------------------------------- fused rotate-on-load (a7)
_FUSED = {}


def run_fused(name, splits=0, rope_style=0):
    key = (name, splits, rope_style)
    if key in _FUSED:
        return _FUSED[key]
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    import paper_2607_28069_gb300 as pic
    wl = generate(SMALL[name], device="cuda", gen_device="cpu")
    path = CacheHitPath(wl, prefill_splits=splits, with_lse=True, rope_style=rope_style)
    path.fused_pass()        # compose + append + fused attention; the cache never sees a document
    torch.cuda.synchronize()
    assert pic.pic_device_status() == (0, 0)
    _FUSED[key] = (wl, path)
    return _FUSED[key]


@pytest.mark.parametrize("name", ["tiny", "llama8b_1layer", "ragged_b3", "gqa7_decode", "d64_g8",
                                  "no_docs", "spans_b2", "spans_d64", "boundary_blocks",
                                  "base_mixed", "base_far_spans", "base_far_d128"])
@pytest.mark.parametrize("splits", [0, 1, 3])
def test_fused_prefill_matches_oracle(cuda_lib, name, splits):
    wl, path = run_fused(name, splits)
    theta = theta_of(wl.spec)
    for layer in range(wl.spec.layers):
        for b in range(wl.spec.batch):
            lay = oracle_layout(wl, b)
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
            (o_ref, lse_ref), _, _ = O.cache_hit_prefill(
                lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), q, k, v, theta,
                return_lse=True)
            o_gpu = f64(path.out[layer, b, :q.shape[0]])
            ok, max_abs, row = attn_close(o_gpu, o_ref)
            assert ok, f"layer {layer} req {b}: err/bound {max_abs:.2f} row-rel {row:.2e}"
            assert np.abs(f64(path.lse[layer, b, :q.shape[0]]) - lse_ref).max() < 5e-2
    # the relocated cache was never written: document slots are still zero
    if wl.spec.docs_per_request:
        lay = oracle_layout(wl, 0)
        t = lay.doc_offset[0]
        s = int(lay.slot_mapping[t])
        assert float(path.k_cache[0].reshape(-1, wl.spec.kv_heads, 16, wl.spec.head_dim)[
            s // 16, :, s % 16].abs().max()) == 0.0


@pytest.mark.parametrize("name", ["ragged_b3", "base_mixed", "base_far_d128"])
def test_fused_interleaved_rope(cuda_lib, name):
    wl, path = run_fused(name, 0, rope_style=1)
    theta = theta_of(wl.spec)
    for b in range(wl.spec.batch):
        lay = oracle_layout(wl, b)
        last = wl.spec.layers - 1
        docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, last)
        o_ref, _, _ = O.cache_hit_prefill(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(),
                                          q, k, v, theta, O.INTERLEAVED)
        ok, max_abs, row = attn_close(f64(path.out[last, b, :q.shape[0]]), o_ref)
        assert ok, (max_abs, row)


@pytest.mark.parametrize("name,rope_style", [("llama8b_1layer", 0), ("ragged_b3", 0),
                                             ("ragged_b3", 1), ("base_mixed", 0),
                                             ("base_far_spans", 1), ("spans_d64", 0),
                                             ("boundary_blocks", 0), ("many_docs", 0),
                                             ("d64_g8", 1), ("no_docs", 0)])
@pytest.mark.parametrize("splits", [0, 1])
def test_fused_equals_materialised(cuda_lib, name, rope_style, splits):
    """Rotate-on-load rotates each document key in shared memory with the
    relocation's own arithmetic, so its outputs equal the materialised
    pass's bit for bit (same split count), while the documents' cache slots
    stay unwritten."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL[name], device="cuda", gen_device="cpu")
    m = CacheHitPath(wl, prefill_splits=splits, with_lse=True, rope_style=rope_style)
    m.ttft_pass()
    f = CacheHitPath(wl, prefill_splits=splits, with_lse=True, rope_style=rope_style)
    f.fused_pass()
    torch.cuda.synchronize()
    import paper_2607_28069_gb300 as pic
    assert pic.pic_device_status() == (0, 0)
    for bb in range(wl.spec.batch):
        tin = int(wl.inline_len[bb])
        assert torch.equal(m.out[:, bb, :tin], f.out[:, bb, :tin]), bb
        assert torch.equal(m.lse[:, bb, :tin], f.lse[:, bb, :tin]), bb


@pytest.mark.gpu
def test_packed_request_upload_gives_identical_results():
    """pack_request_inputs + upload (one host-to-device copy per request)
    must leave the pass's results bit-identical to the unpacked tensors."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL["spans_b2"], device="cuda", gen_device="cpu")
    path = CacheHitPath(wl)
    path.ttft_pass()
    torch.cuda.synchronize()
    ref_out, ref_k = path.out.clone(), path.k_cache.clone()
    host = path.pack_request_inputs()
    path.out.zero_()
    path.k_cache.zero_()
    path.upload(host)
    path.ttft_pass()
    torch.cuda.synchronize()
    for b in range(wl.spec.batch):  # rows past a request's inline tokens are not written
        tin = int(wl.inline_len[b])
        assert torch.equal(path.out[:, b, :tin], ref_out[:, b, :tin]), b
    assert torch.equal(path.k_cache, ref_k)


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["spans_b2", "gqa7_decode", "tiny"])
@pytest.mark.parametrize("graph", [False, True])
def test_served_pass_streams_inputs_and_outputs(cuda_lib, name, graph):
    """served_pass (inputs uploaded and outputs read back per layer, on side
    streams, overlapping the compute) gives the host the outputs of
    ttft_pass bit for bit, run eagerly and replayed from a CUDA graph."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL[name], device="cuda", gen_device="cpu")
    path = CacheHitPath(wl)
    path.ttft_pass()
    torch.cuda.synchronize()
    ref_out, ref_k = path.out.clone(), path.k_cache.clone()
    host = path.pack_request_inputs()
    host_out = torch.zeros(path.out.shape, dtype=path.out.dtype, pin_memory=True)
    up, down = torch.cuda.Stream(), torch.cuda.Stream()
    path.out.zero_()
    path.k_cache.zero_()
    path._request_dev.zero_()        # every input must come from the host mirror
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            path.served_pass(host, host_out, up, down)
        torch.cuda.synchronize()
        path.out.zero_()
        path._request_dev.zero_()
        host_out.zero_()
        g.replay()
    else:
        path.served_pass(host, host_out, up, down)
    torch.cuda.synchronize()
    L, B = wl.spec.layers, wl.spec.batch
    for b in range(B):
        tin = int(wl.inline_len[b])
        assert torch.equal(host_out[:, b, :tin], ref_out[:, b, :tin].cpu())
    assert torch.equal(path.k_cache, ref_k)
    assert L == host_out.shape[0]


@pytest.mark.gpu
@pytest.mark.parametrize("name,rope_style", [("tiny", 0), ("llama8b_1layer", 0), ("ragged_b3", 0),
                                             ("ragged_b3", 1), ("d64_g8", 0), ("no_docs", 0),
                                             ("spans_b2", 0), ("spans_d64", 1),
                                             ("boundary_blocks", 0), ("base_mixed", 0),
                                             ("base_mixed", 1), ("base_far_spans", 0),
                                             ("base_far_d128", 1)])
def test_link_equals_separate_calls(name, rope_style):
    """pic_link (layout + relocation + first-layer append in one launch) gives
    bit-identical layout outputs, caches and prefill outputs to pic_compose,
    pic_relocate and pic_append_inline called in turn."""
    import paper_2607_28069_gb300 as pic
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL[name], device="cuda", gen_device="cpu")
    outs = []
    for linked in (False, True):
        path = CacheHitPath(wl, with_lse=True, rope_style=rope_style)
        path.ttft_pass(linked=linked)
        torch.cuda.synchronize()
        assert pic.pic_device_status() == (0, 0)
        outs.append({k: getattr(path, k).clone() for k in
                     ("doc_offset", "doc_delta", "slot_mapping", "tok_map", "inline_pos", "ctx_len",
                      "k_cache", "v_cache", "out", "lse")})
    for k in ("doc_offset", "doc_delta", "slot_mapping", "tok_map", "inline_pos", "ctx_len",
              "k_cache", "v_cache"):
        assert torch.equal(outs[0][k], outs[1][k]), k
    for b in range(wl.spec.batch):  # out / lse rows past a request's inline tokens are not written
        tin = int(wl.inline_len[b])
        assert torch.equal(outs[0]["out"][:, b, :tin], outs[1]["out"][:, b, :tin]), b
        assert torch.equal(outs[0]["lse"][:, b, :tin], outs[1]["lse"][:, b, :tin]), b


@pytest.mark.gpu
def test_link_reports_bad_document_id():
    """A document id outside the pool is a device-checked error of the link
    launch, as of pic_compose."""
    import paper_2607_28069_gb300 as pic
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL["llama8b_1layer"], device="cuda", gen_device="cpu")
    wl.req_doc_ids[0, 1] = wl.doc_len.numel() + 5
    path = CacheHitPath(wl)
    path.link(0)
    torch.cuda.synchronize()
    code, detail = pic.pic_device_status()
    assert code == 1 and detail == 0
    assert int(path.ctx_len[0]) == -1


def test_per_layer_rotary_tables(cuda_lib):
    """A rotary table per layer (the layer-specific R_l of Eq. 3, e.g. models
    whose layers use different RoPE bases): each layer's relocated keys,
    prefill and decode outputs follow that layer's frequencies, through the
    linked pass and through the fused rotate-on-load pass."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    spec = custom_spec(name="rope_layers", layers=3, q_heads=8, kv_heads=2, head_dim=128,
                       rope_base=1e4, batch=2, pool_docs=4, docs_per_request=3,
                       doc_len=(40, 300), prefix_len=(4, 30), query_len=20, span_len=(0, 5),
                       decode_steps=1)
    thetas = [O.rope_frequencies(128, base) for base in (1e4, 5e5, 1e6)]
    table = torch.tensor(np.stack(thetas), dtype=torch.float64, device="cuda")
    wl = generate(spec, device="cuda", gen_device="cpu")
    # materialised, linked pass + one decode step
    path = CacheHitPath(wl, with_lse=True, layer_inv_freq=table)
    path.ttft_pass()
    path.decode_pass(0)
    # fused rotate-on-load pass
    pathf = CacheHitPath(wl, with_lse=True, layer_inv_freq=table)
    pathf.compose()
    for layer in range(spec.layers):
        pathf.append(layer)
        pathf.attend_fused(layer)
    torch.cuda.synchronize()
    import paper_2607_28069_gb300 as pic
    assert pic.pic_device_status() == (0, 0)
    for layer in range(spec.layers):
        th = thetas[layer]
        for b in range(spec.batch):
            lay = oracle_layout(wl, b)
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
            base = wl.doc_base_pos.cpu().numpy()
            (o_ref, _), K, V = O.cache_hit_prefill(lay, k_docs, v_docs, base, q, k, v, th,
                                                   return_lse=True)
            slots = torch.as_tensor(lay.slot_mapping, device="cuda")
            kc = path.k_cache[layer].reshape(-1, spec.kv_heads, 16, spec.head_dim)
            Kg = f64(kc[slots // 16, :, slots % 16])
            ok, ratio = kv_tolerance_ok(Kg, K)
            assert ok, f"K layer {layer} req {b}: worst err/bound {ratio:.3f}"
            if layer > 0:  # the layer's own table, not layer 0's
                K0, _ = O.dense_context(lay, k_docs, v_docs, base, k, v, thetas[0])
                assert not kv_tolerance_ok(Kg, K0)[0]
            tin = q.shape[0]
            for pp in (path, pathf):
                ok, max_abs, row = attn_close(f64(pp.out[layer, b, :tin]), o_ref)
                assert ok, f"layer {layer} req {b}: err/bound {max_abs:.2f} row-rel {row:.2e}"
            o_dec, _, _ = O.decode_step(K, V, f64(wl.q_dec[0, layer, b]), f64(wl.k_dec[0, layer, b]),
                                        f64(wl.v_dec[0, layer, b]), lay.ctx_len, th)
            ok, max_abs, row = attn_close(f64(path.dec_out[layer, b]), o_dec)
            assert ok, f"decode layer {layer} req {b}: {max_abs:.2e} {row:.2e}"


@pytest.mark.parametrize("name,rows", [("spans_b2", "query"), ("llama8b_1layer", "query"),
                                       ("spans_d64", "query"), ("boundary_blocks", "query"),
                                       ("spans_b2", "inline"), ("boundary_blocks", "inline"),
                                       ("many_docs", "query")])
def test_attention_deviation_matches_oracle(cuda_lib, name, rows):
    """D_r(A, B) of the diagnostic on the GPU against the oracle, with A = the
    relocated cache and B = the same documents copied at their compiled
    positions (no re-rotation: every delta 0), over the paper's pre / int
    regions and a four-region split.  rows="inline" takes every inline token
    as a query row: prefix and span rows come before later documents, whose
    keys they do not see."""
    import paper_2607_28069_gb300 as pic
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL[name], device="cuda", gen_device="cpu")
    spec = wl.spec
    A = CacheHitPath(wl, with_lse=True)
    Bp = CacheHitPath(wl, with_lse=True)
    A.compose()
    A.relocate()
    Bp.compose()
    pic.pic_relocate_mapped(Bp.geom, wl.k_pool, wl.v_pool, Bp.tok_map, torch.zeros_like(Bp.doc_delta),
                     Bp.slot_mapping, wl.num_pages, Bp.k_cache, Bp.v_cache, 0, spec.layers)
    theta = theta_of(spec)
    if rows == "query":
        query_len = torch.full((spec.batch,), spec.query_len, dtype=torch.int32, device="cuda")
    else:
        query_len = wl.inline_len.to(torch.int32).clone()
    for edges in ((0.0, 0.1, 0.9), (0.0, 0.25, 0.5, 0.75, 1.0)):
        R = len(edges) - 1
        for layer in range(spec.layers):
            for p in (A, Bp):
                p.append(layer)
                p.attend(layer)
            sums = torch.empty((spec.batch, R), dtype=torch.float64, device="cuda")
            counts = torch.empty((spec.batch, R), dtype=torch.int64, device="cuda")
            pic.pic_attention_deviation(A.geom, layer, A.inline_pos, wl.inline_len, query_len,
                                        wl.req_doc_ids, wl.doc_len, A.doc_offset, A.slot_mapping,
                                        wl.num_pages, A.k_cache, Bp.k_cache,
                                        A.lse[layer], Bp.lse[layer], A.ws_prefill, sums, counts,
                                        edges)
            torch.cuda.synchronize()
            assert pic.pic_device_status() == (0, 0)
            for b in range(spec.batch):
                lay = oracle_layout(wl, b)
                docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
                base = wl.doc_base_pos.cpu().numpy()
                Ka, _ = O.dense_context(lay, k_docs, v_docs, base, k, v, theta, storage="bf16")
                Kb = Ka.copy()       # B: every document occurrence as compiled (delta 0)
                for i, kd in enumerate(k_docs):
                    Kb[lay.doc_offset[i]:lay.doc_offset[i] + kd.shape[0]] = kd
                tq = int(query_len[b])
                qp = lay.inline_pos[-tq:]
                qr = O.round_bf16(O.rotary(q[-tq:], qp[:, None], theta))
                lens = [int(wl.doc_len[dd]) for dd in docs]
                s_ref, c_ref = O.attention_deviation(qr, qp, Ka, Kb, lay, lens, edges)
                assert np.array_equal(counts[b].cpu().numpy(), c_ref), (layer, b)
                got = sums[b].cpu().numpy()
                np.testing.assert_allclose(got, s_ref, rtol=2e-2, atol=1e-6 * c_ref.max())
                assert (s_ref > 0).all()


@pytest.mark.gpu
@pytest.mark.parametrize("splits", [1, 0])
def test_prefill_output_into_pinned_host_memory(cuda_lib, splits):
    """pic_attend_prefill with `out` in page-locked host memory: the kernels
    (the attention epilogue with one split, the merge kernel with several)
    store the rows there, bit for bit the rows they store on the device."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL["spans_b2"], device="cuda", gen_device="cpu")
    path = CacheHitPath(wl, prefill_splits=splits)
    path.ttft_pass()
    host = torch.zeros(path.out[0].shape, dtype=path.out.dtype, pin_memory=True)
    for layer in range(wl.spec.layers):
        path.append(layer)      # the workspace holds one layer's rotated queries
        path.attend(layer)
        host.zero_()
        path.attend(layer, out=host)
        torch.cuda.synchronize()
        for b in range(wl.spec.batch):
            tin = int(wl.inline_len[b])
            assert torch.equal(host[b, :tin], path.out[layer, b, :tin].cpu())


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["gqa7_decode", "g16_decode", "spans_b2"])
def test_decode_split_count_invariance(cuda_lib, name):
    """Every split of the key range gives the same decode output: the LSE
    merge is exact up to rounding, so outputs for 1, 3 and the automatic
    number of splits agree within 1e-3 (max-abs)."""
    outs = []
    for splits in (1, 3, 0):
        wl, path, dec = run_path(name, decode_splits=splits)
        outs.append([d[0].float() for d in dec])
    for s in range(len(outs[0])):
        for other in outs[1:]:
            diff = (other[s] - outs[0][s]).abs().max().item()
            assert diff <= 1e-3, f"{name} step {s}: split-count difference {diff:.2e}"


@pytest.mark.gpu
@pytest.mark.parametrize("name,splits", [("tiny", 0), ("llama8b_1layer", 0), ("llama8b_1layer", 5),
                                         ("gqa7_decode", 0), ("d64_g8", 0), ("long_prefix", 0),
                                         ("no_docs", 0), ("boundary_blocks", 0)])
def test_single_visible_key_returns_its_value_bit_exact(cuda_lib, name, splits):
    """The first prefix token sees only itself (position 0), so its softmax
    has one term, p = 1, and its output is its own value, bit for bit: every
    layer and query head, with and without key splits."""
    wl, path, _ = run_path(name, prefill_splits=splits)
    G = wl.spec.q_heads // wl.spec.kv_heads
    for b in range(wl.spec.batch):
        if int(wl.prefix_len[b]) < 1:
            continue
        out = path.out[:, b, 0]                                    # [L][Hq][d]
        v0 = wl.v_inline[:, b, 0].repeat_interleave(G, dim=1)      # [L][Hq][d]
        assert torch.equal(out, v0), f"request {b}: {(out.float() - v0.float()).abs().max():.2e}"


@pytest.mark.gpu
@pytest.mark.parametrize("splits", [1, 0])
def test_zero_keys_give_the_mean_of_visible_values(cuda_lib, splits):
    """With every key zero the scores are all zero and the softmax uniform:
    each output row is the mean of the values at or before its position
    (computed here in fp64 from the inputs), through spans, documents and
    the split merge."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    wl = generate(SMALL["spans_b2"], device="cuda", gen_device="cpu")
    wl.k_pool.zero_()
    wl.k_inline.zero_()
    path = CacheHitPath(wl, prefill_splits=splits)
    path.ttft_pass()
    torch.cuda.synchronize()
    theta = theta_of(wl.spec)
    G = wl.spec.q_heads // wl.spec.kv_heads
    for layer in range(wl.spec.layers):
        for b in range(wl.spec.batch):
            lay = oracle_layout(wl, b)
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
            _, V = O.dense_context(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), k, v, theta)
            pos = np.asarray(lay.inline_pos)
            csum = np.cumsum(V, axis=0)                               # [ctx][Hkv][d]
            ref = csum[pos] / (pos + 1)[:, None, None]                # [T][Hkv][d]
            ref = np.repeat(ref, G, axis=1)                           # [T][Hq][d]
            ok, max_abs, row = attn_close(f64(path.out[layer, b, :len(pos)]), ref)
            assert ok, f"layer {layer} req {b}: err/bound {max_abs:.2f} row-rel {row:.2e}"
