"""Each entry point of the C ABI on its own: arguments as the paper states the
problem (per-document blocks, base and target positions, the inline tokens'
projections and positions), results against the oracle.

* pic_relocate with placements pic_compose would never produce (documents
  out of order, gaps between them, a document listed twice);
* pic_attend_prefill given the projections, over a cache that only
  pic_relocate filled (no pic_compose, pic_append_inline or pic_link);
* pic_relocate and pic_relocate_mapped give bit-identical caches;
* overlapping targets are a device-checked error.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2607_28069_gb300.workloads import custom_spec, generate
from tests.helpers import attn_close, f64, kv_tolerance_ok, oracle_layout, request_inputs, theta_of

pytestmark = pytest.mark.gpu

SPEC = custom_spec(name="boundary", layers=2, q_heads=16, kv_heads=4, head_dim=128,
                   rope_base=5e5, batch=2, pool_docs=5, docs_per_request=4, doc_len=(20, 260),
                   prefix_len=(5, 40), query_len=33, base_pos=(0, 3000))


def _geom(spec, rope_style=0):
    import paper_2607_28069_gb300 as pic
    return pic.Geometry(spec.layers, spec.q_heads, spec.kv_heads, spec.head_dim, spec.rope_base,
                        rope_style=rope_style)


def _cache(spec, num_pages):
    shape = (spec.layers, num_pages, spec.kv_heads, 16, spec.head_dim)
    return (torch.zeros(shape, dtype=torch.bfloat16, device="cuda"),
            torch.zeros(shape, dtype=torch.bfloat16, device="cuda"))


@pytest.mark.parametrize("rope_style", [0, 1])
def test_relocate_places_documents_anywhere(cuda_lib, rope_style):
    """Documents moved to arbitrary targets (reversed order, gaps, one pool
    document listed twice): every slot of every document holds
    R(target - base) k (Eq. 3) within the key bar, and its value bit for bit;
    slots outside the documents stay untouched."""
    import paper_2607_28069_gb300 as pic
    spec = SPEC
    wl = generate(spec, device="cuda", gen_device="cpu")
    lens = wl.doc_len.cpu().numpy()
    base = wl.doc_base_pos.cpu().numpy()
    starts = wl.doc_token_start.cpu().numpy()
    # request 0: pool docs 3, 1, 4 with gaps of 7 and 40 positions, from 11;
    # request 1: doc 2 twice and doc 0, from 0, no gaps
    orders = [[3, 1, 4], [2, 0, 2]]
    targets = []
    for b, order in enumerate(orders):
        t, row = (11, []) if b == 0 else (0, [])
        gaps = [7, 40, 0] if b == 0 else [0, 0, 0]
        for d, gp in zip(order, gaps):
            row.append(t)
            t += int(lens[d]) + gp
        targets.append(row)
    need = max(tg[-1] + int(lens[o[-1]]) for tg, o in zip(targets, orders))
    pages = -(-need // 16)
    rng = np.random.default_rng(7)
    perm = rng.permutation(2 * pages).astype(np.int32)
    bt = torch.tensor(perm.reshape(2, pages), device="cuda")
    ids = torch.tensor(orders, dtype=torch.int32, device="cuda")
    tgt = torch.tensor(targets, dtype=torch.int32, device="cuda")
    ndocs = torch.tensor([3, 3], dtype=torch.int32, device="cuda")
    kc, vc = _cache(spec, 2 * pages)
    geom = _geom(spec, rope_style)
    pic.pic_relocate(geom, wl.k_pool, wl.v_pool, wl.doc_token_start, wl.doc_len,
                     wl.doc_base_pos, ids, ndocs, tgt, bt, 2 * pages, kc, vc, 0, spec.layers)
    torch.cuda.synchronize()
    assert pic.pic_device_status() == (0, 0)
    theta = theta_of(spec)
    style = O.INTERLEAVED if rope_style else O.HALF
    written = np.zeros((2, pages * 16), bool)
    for layer in range(spec.layers):
        for b in range(2):
            for d, t0 in zip(orders[b], targets[b]):
                n = int(lens[d])
                t = t0 + np.arange(n)
                slot = perm.reshape(2, pages)[b][t // 16].astype(np.int64) * 16 + t % 16
                s = torch.as_tensor(slot, device="cuda")
                Kg = f64(kc[layer][s // 16, :, s % 16])
                Vg = f64(vc[layer][s // 16, :, s % 16])
                kraw = f64(wl.k_pool[layer, starts[d]:starts[d] + n])
                Kr = O.rerotate_key(kraw, (base[d] + np.arange(n))[:, None], t[:, None], theta,
                                    style)
                ok, ratio = kv_tolerance_ok(Kg, Kr)
                assert ok, f"layer {layer} req {b} doc {d}: err/bound {ratio:.2f}"
                assert np.array_equal(Vg, f64(wl.v_pool[layer, starts[d]:starts[d] + n]))
                written[b, t] = True
    # positions in the gaps were not written
    for b in range(2):
        free = np.nonzero(~written[b, :need])[0]
        if free.size:
            slot = perm.reshape(2, pages)[b][free // 16].astype(np.int64) * 16 + free % 16
            s = torch.as_tensor(slot, device="cuda")
            assert float(kc[:, s // 16, :, s % 16].abs().max()) == 0.0


def test_prefill_on_its_own_over_a_relocated_cache(cuda_lib):
    """pic_relocate (targets from the oracle's layout) then pic_attend_prefill
    given the inline projections and positions: no pic_compose, no separate
    append.  Outputs against the oracle's cache-hit prefill."""
    import paper_2607_28069_gb300 as pic
    spec = SPEC
    wl = generate(spec, device="cuda", gen_device="cpu")
    B = spec.batch
    lays = [oracle_layout(wl, b) for b in range(B)]
    md = wl.req_doc_ids.shape[1]
    tgt = torch.tensor([lay.doc_offset + [0] * (md - len(lay.doc_offset)) for lay in lays],
                       dtype=torch.int32, device="cuda")
    ipos = torch.full((B, wl.tin_max), -1, dtype=torch.int32, device="cuda")
    for b, lay in enumerate(lays):
        ipos[b, :len(lay.inline_pos)] = torch.as_tensor(lay.inline_pos, dtype=torch.int32)
    geom = _geom(spec)
    kc, vc = _cache(spec, wl.num_pages)
    pic.pic_relocate(geom, wl.k_pool, wl.v_pool, wl.doc_token_start, wl.doc_len,
                     wl.doc_base_pos, wl.req_doc_ids, wl.req_num_docs, tgt, wl.block_table,
                     wl.num_pages, kc, vc, 0, spec.layers)
    ws = torch.empty(pic.pic_prefill_workspace_size(geom, B, wl.tin_max, wl.max_ctx, 0),
                     dtype=torch.uint8, device="cuda")
    out = torch.zeros((spec.layers, B, wl.tin_max, spec.q_heads, spec.head_dim),
                      dtype=torch.bfloat16, device="cuda")
    for layer in range(spec.layers):
        pic.pic_attend_prefill(geom, layer, ipos, wl.inline_len, wl.max_ctx, wl.block_table,
                               wl.num_pages, kc, vc, out[layer], None, 0, ws,
                               q=wl.q_inline[layer], k_new=wl.k_inline[layer],
                               v_new=wl.v_inline[layer])
    torch.cuda.synchronize()
    assert pic.pic_device_status() == (0, 0)
    theta = theta_of(spec)
    for layer in range(spec.layers):
        for b in range(B):
            docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
            o_ref, _, _ = O.cache_hit_prefill(lays[b], k_docs, v_docs,
                                              wl.doc_base_pos.cpu().numpy(), q, k, v, theta)
            ok, ratio, row = attn_close(f64(out[layer, b, :q.shape[0]]), o_ref)
            assert ok, f"layer {layer} req {b}: err/bound {ratio:.2f} row-rel {row:.2e}"


@pytest.mark.parametrize("name", ["ragged_b3", "spans_d64", "boundary_blocks", "base_mixed"])
def test_relocate_forms_are_bit_identical(cuda_lib, name):
    """The per-document form (targets = pic_compose's doc_offset) and the
    map form write the same caches, bit for bit."""
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    from tests.test_gpu_parity import SMALL
    wl = generate(SMALL[name], device="cuda", gen_device="cpu")
    a, m = CacheHitPath(wl), CacheHitPath(wl)
    a.compose()
    a.relocate()
    m.compose()
    m.relocate_mapped()
    torch.cuda.synchronize()
    assert torch.equal(a.k_cache, m.k_cache) and torch.equal(a.v_cache, m.v_cache)


def test_relocate_reports_overlapping_targets(cuda_lib):
    import paper_2607_28069_gb300 as pic
    spec = SPEC
    wl = generate(spec, device="cuda", gen_device="cpu")
    lens = wl.doc_len.cpu().numpy()
    ids = torch.tensor([[0, 1]], dtype=torch.int32, device="cuda")
    t1 = int(lens[0]) - 1                      # doc 1 starts on doc 0's last position
    tgt = torch.tensor([[0, t1]], dtype=torch.int32, device="cuda")
    pages = -(-(t1 + int(lens[1])) // 16)
    bt = torch.arange(pages, dtype=torch.int32, device="cuda")[None]
    kc, vc = _cache(spec, pages)
    pic.pic_relocate(_geom(spec), wl.k_pool, wl.v_pool, wl.doc_token_start, wl.doc_len,
                     wl.doc_base_pos, ids, torch.tensor([2], dtype=torch.int32, device="cuda"),
                     tgt, bt, pages, kc, vc, 0, spec.layers)
    code, detail = pic.pic_device_status()
    assert code == 7 and detail == 0
    # a block table one page short is reported too
    pic.pic_relocate(_geom(spec), wl.k_pool, wl.v_pool, wl.doc_token_start, wl.doc_len,
                     wl.doc_base_pos, ids[:, :1], torch.tensor([1], dtype=torch.int32,
                                                                device="cuda"),
                     torch.tensor([[16]], dtype=torch.int32, device="cuda"),
                     bt[:, :max(1, -(-int(lens[0]) // 16))], pages, kc, vc, 0, spec.layers)
    code, _ = pic.pic_device_status()
    assert code == 5


def test_launch_probe_runs_a_dependent_chain(cuda_lib):
    """The measurement aid launches a chain of empty dependent kernels with
    the attention's shape (384 threads, 230 KB of shared memory) and rejects
    a block above 1024 threads."""
    import paper_2607_28069_gb300 as pic
    shapes = [((268, 1, 1), 256, 0), ((144, 1, 1), 384, 230912), ((768, 1, 1), 256, 0)]
    pic.pic_launch_probe(shapes)
    torch.cuda.synchronize()
    with pytest.raises(pic.PicError):
        pic.pic_launch_probe([((1, 1, 1), 2048, 0)])
