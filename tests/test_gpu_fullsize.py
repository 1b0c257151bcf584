"""Parity at full size: the 32-layer batch-8 Llama-3-8B workload, the 28-layer
batch-16 decode workload and the 4 x ~139k-token stress workload, generated
and run as bench.py times them (the linked TTFT pass with the automatic split
counts; one decode step), checked against the oracle on sampled outputs the
oracle computes one by one:

* the layout and slot map of every request, in full (bit-exact);
* the stitched cache of two sampled layers (every document and inline
  position of sampled requests, read back through the slots): K within the
  relocated-key bar, V bit-exact;
* the prefill attention of sampled (request, layer) pairs for 64 sampled
  inline rows including the last one (every head; one kv-head group for the
  ~139k-token contexts);
* for the decode workload, one decode step of a sampled request and layer;
* for the 32-layer batch-8 and the stress workloads, the fused rotate-on-load
  attention of the same two layers (their caches cleared first, so that the
  documents can only come from the pool), on the same sampled rows of one
  kv-head group per sampled request.

Each case frees its device memory when it ends.
"""
import dataclasses
import gc

import numpy as np
import pytest
import torch

import oracle as O
from paper_2607_28069_gb300.workloads import WORKLOADS, generate
from tests.helpers import (attn_close, f64, kv_tolerance_ok, oracle_layout, request_inputs,
                           theta_of)

pytestmark = pytest.mark.gpu

FULL = ["llama8b_32layer_b8", "decode_28layer_b16", "stress_128k_b4"]


def _run(name):
    from paper_2607_28069_gb300.pipeline import CacheHitPath
    import paper_2607_28069_gb300 as pic
    spec = WORKLOADS[name]
    if spec.decode_steps > 1:
        spec = dataclasses.replace(spec, decode_steps=1)
    wl = generate(spec, device="cuda", gen_device="cuda")
    path = CacheHitPath(wl, with_lse=False)
    path.ttft_pass()
    if wl.q_dec is not None:
        path.decode_pass(0)
    torch.cuda.synchronize()
    code, detail = pic.pic_device_status()
    assert code == 0, f"device status {code} detail {detail}"
    return wl, path


def _check_layout(wl, path):
    off, dl = path.doc_offset.cpu().numpy(), path.doc_delta.cpu().numpy()
    slots, ipos = path.slot_mapping.cpu().numpy(), path.inline_pos.cpu().numpy()
    ctx = path.ctx_len.cpu().numpy()
    for b in range(wl.spec.batch):
        lay = oracle_layout(wl, b)
        m = len(lay.doc_ids)
        assert ctx[b] == lay.ctx_len
        assert list(off[b, :m]) == lay.doc_offset and list(dl[b, :m]) == lay.doc_delta
        assert np.array_equal(slots[b, :lay.ctx_len], lay.slot_mapping)
        assert np.array_equal(ipos[b, :len(lay.inline_pos)], lay.inline_pos)


def _dense(wl, b, layer, theta):
    lay = oracle_layout(wl, b)
    docs, k_docs, v_docs, q, k, v = request_inputs(wl, b, layer)
    K, V = O.dense_context(lay, k_docs, v_docs, wl.doc_base_pos.cpu().numpy(), k, v, theta)
    return lay, q, K, V


def _check_cache(wl, path, b, layer, lay, K, V):
    spec = wl.spec
    slots = torch.as_tensor(lay.slot_mapping, device="cuda")
    kc = path.k_cache[layer].reshape(-1, spec.kv_heads, spec.page_size, spec.head_dim)
    vc = path.v_cache[layer].reshape(-1, spec.kv_heads, spec.page_size, spec.head_dim)
    Kg = f64(kc[slots // spec.page_size, :, slots % spec.page_size])
    Vg = f64(vc[slots // spec.page_size, :, slots % spec.page_size])
    ok, ratio = kv_tolerance_ok(Kg, K)
    assert ok, f"K layer {layer} req {b}: worst err/bound {ratio:.3f}"
    assert np.array_equal(Vg, V), f"V layer {layer} req {b} must be a bit copy"


def _check_attention(wl, path, b, layer, lay, q, K, V, theta, rng, kv_groups):
    spec = wl.spec
    G = spec.q_heads // spec.kv_heads
    tin = q.shape[0]
    rows = np.sort(np.concatenate([rng.choice(tin - 1, size=min(63, tin - 1), replace=False),
                                   [tin - 1]]))
    qp = np.asarray(lay.inline_pos)[rows]
    qr = O.rotary(q[rows], qp[:, None], theta)
    out = f64(path.out[layer, b, torch.as_tensor(rows, device="cuda")])
    for g in kv_groups:
        heads = slice(g * G, (g + 1) * G)
        o_ref = O.attention(qr[:, heads], qp, K[:, g:g + 1], V[:, g:g + 1])
        ok, max_abs, row = attn_close(out[:, heads], o_ref)
        assert ok, f"layer {layer} req {b} kv group {g}: err/bound {max_abs:.2f} row-rel {row:.2e}"


def _check_decode(wl, path, b, layer, lay, K, V, theta):
    o_ref, _, _ = O.decode_step(K, V, f64(wl.q_dec[0, layer, b]), f64(wl.k_dec[0, layer, b]),
                                f64(wl.v_dec[0, layer, b]), lay.ctx_len, theta)
    ok, max_abs, row = attn_close(f64(path.dec_out[layer, b]), o_ref)
    assert ok, f"decode layer {layer} req {b}: err/bound {max_abs:.2f} row-rel {row:.2e}"


FUSED = ["llama8b_32layer_b8", "stress_128k_b4"]


def _check_fused(wl, path, layers, reqs, theta):
    """Fused rotate-on-load attention at full size: the sampled layers'
    caches are zeroed and refilled with the inline tokens only, so every
    document key and value must come from the pool, rotated by -delta on
    the query side."""
    import paper_2607_28069_gb300 as pic
    spec = wl.spec
    rng = np.random.default_rng(28069)
    for layer in layers:
        path.k_cache[layer].zero_()
        path.v_cache[layer].zero_()
        path.out[layer].zero_()
        path.append(layer)
        path.attend_fused(layer)
        torch.cuda.synchronize()
        code, detail = pic.pic_device_status()
        assert code == 0, f"device status {code} detail {detail}"
        for b in reqs:
            lay, q, K, V = _dense(wl, b, layer, theta)
            groups = [int(rng.integers(spec.kv_heads))]
            _check_attention(wl, path, b, layer, lay, q, K, V, theta, rng, groups)
            del K, V


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled_parity(cuda_lib, name):
    wl, path = _run(name)
    try:
        spec = wl.spec
        theta = theta_of(spec)
        rng = np.random.default_rng(2607)
        _check_layout(wl, path)
        long_ctx = spec.docs_per_request * spec.doc_len[1] > 100_000
        layers = [0, int(rng.integers(1, spec.layers))]
        n_req = 1 if long_ctx else 2
        reqs = [0] + [int(x) for x in rng.choice(np.arange(1, spec.batch), n_req - 1,
                                                  replace=False)]
        kv_groups = [int(rng.integers(spec.kv_heads))] if long_ctx else range(spec.kv_heads)
        for layer in layers:
            for b in reqs:
                lay, q, K, V = _dense(wl, b, layer, theta)
                _check_cache(wl, path, b, layer, lay, K, V)
                _check_attention(wl, path, b, layer, lay, q, K, V, theta, rng, kv_groups)
                if wl.q_dec is not None:
                    _check_decode(wl, path, b, layer, lay, K, V, theta)
                del K, V
        if name in FUSED:
            _check_fused(wl, path, layers, reqs, theta)
    finally:
        del path, wl
        gc.collect()
        torch.cuda.empty_cache()
