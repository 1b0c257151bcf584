"""Test-side glue: turn a workload into oracle inputs and compare results.

Test infrastructure only (imports the oracle).  Nothing here does the
method's arithmetic: it slices inputs and calls ``oracle``.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle as O


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def request_inputs(wl, b: int, layer: int):
    """Oracle inputs of request b, layer `layer` (numpy float64 / int)."""
    docs = wl.meta["docs"][b]
    starts = wl.doc_token_start.cpu().numpy()
    lens = wl.doc_len.cpu().numpy()
    k_docs = [f64(wl.k_pool[layer, starts[d]:starts[d] + lens[d]]) for d in docs]
    v_docs = [f64(wl.v_pool[layer, starts[d]:starts[d] + lens[d]]) for d in docs]
    tin = int(wl.inline_len[b])
    q = f64(wl.q_inline[layer, b, :tin])
    k = f64(wl.k_inline[layer, b, :tin])
    v = f64(wl.v_inline[layer, b, :tin])
    return docs, k_docs, v_docs, q, k, v


def oracle_layout(wl, b: int):
    spec = wl.spec
    return O.compose_layout(wl.doc_len.cpu().numpy(), wl.doc_base_pos.cpu().numpy(),
                            wl.meta["docs"][b], int(wl.prefix_len[b]), spec.query_len,
                            wl.block_table[b].cpu().numpy(), spec.page_size,
                            span_len=wl.meta["spans"][b])


def theta_of(spec):
    return O.rope_frequencies(spec.head_dim, spec.rope_base)


def kv_tolerance_ok(gpu: np.ndarray, ref: np.ndarray, rel: float = 4e-3):
    """Relocated-key bar: per element |g - r| <= rel * max(|r|, 2^-8 * rowmax),
    and per (token, head) row relative L2 <= rel.  Returns (ok, worst_ratio)."""
    rowmax = np.abs(ref).max(axis=-1, keepdims=True)
    bound = rel * np.maximum(np.abs(ref), rowmax * 2.0 ** -8)
    err = np.abs(gpu - ref)
    ratio = float((err / np.maximum(bound, 1e-30)).max()) if err.size else 0.0
    l2 = np.linalg.norm(gpu - ref, axis=-1) / np.maximum(np.linalg.norm(ref, axis=-1), 1e-30)
    return ratio <= 1.0 and float(l2.max(initial=0.0)) <= rel, ratio


def half_ulp_bf16(x: np.ndarray) -> np.ndarray:
    """Half the spacing of bfloat16 values at |x| (8 significant bits): for
    2^e <= |x| < 2^(e+1) the spacing is 2^(e-7); below the normal range the
    subnormal spacing 2^-133."""
    a = np.maximum(np.abs(np.asarray(x, np.float64)), 2.0 ** -126)
    e = np.floor(np.log2(a))
    return 2.0 ** (e - 8)


def attn_close(gpu: np.ndarray, ref: np.ndarray, abs_tol=1e-2, row_rel=2e-2):
    """Attention bar: per element |g - r| <= 1e-2 + half a bf16 ulp at
    max(|g|, |r|), and per-row relative L2 <= 2e-2.  The output is stored in
    bf16, so an exact fp32 result still moves by up to half an ulp of the
    stored value when rounded; the 1e-2 is the error allowed on top of that
    rounding (it dominates for |o| < 4).  The ulp is taken at the larger of
    the two magnitudes because the stored value may round up into the next
    binade.  Returns (ok, worst |g - r| / bound, worst row rel-L2); the first
    is <= 1 when the elements pass."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(gpu - ref)
    bound = abs_tol + half_ulp_bf16(np.maximum(np.abs(gpu), np.abs(ref)))
    ratio = float((err / bound).max(initial=0.0))
    l2 = np.linalg.norm(gpu - ref, axis=-1) / np.maximum(np.linalg.norm(ref, axis=-1), 1e-6)
    worst = float(l2.max(initial=0.0))
    return (ratio <= 1.0 and worst <= row_rel), ratio, worst
