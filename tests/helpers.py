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


def attn_close(gpu: np.ndarray, ref: np.ndarray, abs_tol=1e-2, row_rel=2e-2):
    """Attention bar: |g - r| <= 1e-2 * max(1, max|r_row|) and per-row relative
    L2 <= 2e-2.  The output is bf16, so rows with |o| > 1 (short contexts)
    carry proportionally more rounding; for |o| <= 1 the bar is max-abs 1e-2.
    Returns (ok, worst max-abs over rows scaled to the bar, worst row rel-L2)."""
    err = np.abs(gpu - ref)
    scale = np.maximum(1.0, np.abs(ref).max(axis=-1, keepdims=True))
    max_abs = float((err / scale).max(initial=0.0))
    l2 = np.linalg.norm(gpu - ref, axis=-1) / np.maximum(np.linalg.norm(ref, axis=-1), 1e-6)
    worst = float(l2.max(initial=0.0))
    return (max_abs <= abs_tol and worst <= row_rel), max_abs, worst
