"""Plain, slow CPU oracle for the SemPIC cache-hit path.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` use it.  It shares
no code with the CUDA library (``paper_2607_28069_gb300/csrc``) and imports
nothing from the package.

Everything is float64 numpy.  Inputs are the exact values of the bf16 tensors
the GPU path receives (bf16 -> float is exact), so both sides start from the
same numbers; the oracle then does the mathematics without any rounding to
bf16 or fp32.

What the path computes (SemPIC, "Background: Position-Independent Caching" and
"Cache-hit serving"; appendix "Position-Independent Linking"):

1. ``compose_layout``   the link operator R assigns final logical positions in
                         the canonical order P, D_1, S_1, ..., D_m, S_m, Q
                         (Eqs. 1-2; the post-document inline spans S_k may be
                         empty) and
                         builds the token-level map from logical positions to
                         physical paged-cache slots (appendix, "Logical Layout
                         and Re-Rotation").
2. ``rerotate_key``      moves a key created at position a to position b with
                         k~_b = R(b) R(a)^-1 k_a (Eq. 3); values are copied
                         as they are.
3. ``rotary``            the rotary transform R(p) itself (RoPE, cited by the
                         paper as the positional scheme of the evaluated
                         decoders) used for the inline tokens' own keys and
                         queries at their logical positions.
4. ``attention``         the unchanged Reader's softmax attention with GQA head
                         sharing under the frontier causal mask: a token at
                         logical position p sees exactly the keys at logical
                         positions <= p (appendix, "frontier causal mask").
5. ``cache_hit_prefill`` / ``decode_step``  the whole path for one request and
                         one layer: layout, re-rotation, inline RoPE, attention
                         over the stitched context, then ordinary decoding.

Readings where the paper is silent:
* R(p) pairs element i with i + d/2 ("half-split", the convention of the
  Llama/Qwen decoders the paper evaluates); ``style="interleaved"`` pairs
  (2i, 2i+1).  Frequencies theta_i = base^(-2i/d), no scaling, one table for
  all layers.
* Softmax scale 1/sqrt(d); q head h reads kv head floor(h / G), G = Hq / Hkv.
* Pages are filled contiguously in logical order:
  slot(t) = block_table[t // page_size] * page_size + t % page_size.

Parity pins for every function live in ``tests/test_oracle_pins.py``; no
function here is unpinned.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

HALF = "half"
INTERLEAVED = "interleaved"


# --------------------------------------------------------------------------
# bf16 storage (the paper executes in bfloat16: the stitched cache holds bf16
# keys and values, and the Reader consumes bf16 queries)
# --------------------------------------------------------------------------
def round_bf16(x) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 value, ties to even.

    bfloat16 keeps 8 significant bits and the float32 exponent range.  For a
    normal value x = m * 2^e (0.5 <= |m| < 1), the kept significand is
    rint(m * 2^8) (np.rint rounds half to even); below 2^-126 the spacing is
    the fixed subnormal step 2^-133.  Results beyond the largest finite bf16
    become infinities; NaN stays NaN.
    """
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    out = np.ldexp(np.rint(m * 256.0), e - 8)
    tiny = np.abs(x) < 2.0 ** -126
    out = np.where(tiny, np.rint(x * 2.0 ** 133) * 2.0 ** -133, out)
    bf16_max = (2.0 - 2.0 ** -7) * 2.0 ** 127
    out = np.where(np.abs(out) > bf16_max, np.copysign(np.inf, x), out)
    return np.where(np.isfinite(x), out, x)


def _store(x, storage):
    return round_bf16(x) if storage == "bf16" else x


# --------------------------------------------------------------------------
# Rotary transform R(p) and the re-rotation of Eq. 3
# --------------------------------------------------------------------------
def rope_frequencies(head_dim: int, base: float) -> np.ndarray:
    """theta_i = base^(-2i/d) for i < d/2, in float64 (RoPE frequencies)."""
    if head_dim % 2:
        raise ValueError("head_dim must be even")
    i = np.arange(head_dim // 2, dtype=np.float64)
    return np.power(np.float64(base), -2.0 * i / head_dim)


def _pair_index(head_dim: int, style: str):
    """Indices (first, second) of the d/2 rotated pairs."""
    half = head_dim // 2
    if style == HALF:
        return np.arange(half), np.arange(half) + half
    if style == INTERLEAVED:
        return 2 * np.arange(half), 2 * np.arange(half) + 1
    raise ValueError(f"unknown rope style {style!r}")


def rotary(x: np.ndarray, pos, theta: np.ndarray, style: str = HALF) -> np.ndarray:
    """R(pos) x: rotate every pair of ``x`` by the angle pos * theta_i.

    ``x`` has shape [..., d]; ``pos`` is a scalar or broadcasts against
    x.shape[:-1].  For a pair (u, w) with angle phi:
        u' = u cos(phi) - w sin(phi),   w' = u sin(phi) + w cos(phi).
    The angle is formed and evaluated in float64.
    """
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    first, second = _pair_index(d, style)
    pos = np.asarray(pos, dtype=np.float64)
    phi = pos[..., None] * theta  # [..., d/2]
    c, s = np.cos(phi), np.sin(phi)
    u, w = x[..., first], x[..., second]
    out = np.empty(np.broadcast_shapes(x.shape, phi.shape[:-1] + (d,)), dtype=np.float64)
    out[..., first] = u * c - w * s
    out[..., second] = u * s + w * c
    return out


def rerotate_key(k: np.ndarray, a, b, theta: np.ndarray, style: str = HALF) -> np.ndarray:
    """Eq. 3: k~_b = R(b) R(a)^-1 k_a, written as the two rotations it names.

    R(a)^-1 is the rotation by -a (rotations are orthogonal), then R(b) is
    applied.  Only keys go through here; values keep their cached numbers.
    """
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return rotary(rotary(k, -a, theta, style), b, theta, style)


# --------------------------------------------------------------------------
# Link operator: logical layout and physical slots
# --------------------------------------------------------------------------
@dataclass
class RequestLayout:
    """Logical layout of one request (canonical order P, D_1, S_1, ..., D_m, S_m, Q)."""

    prefix_len: int
    doc_ids: list
    doc_offset: list           # first logical position of each doc, in order
    doc_delta: list            # target minus base position of each doc
    query_start: int
    query_len: int
    ctx_len: int
    slot_mapping: np.ndarray = field(repr=False)   # [ctx_len] int64
    inline_pos: np.ndarray = field(repr=False)     # prefix, span and query positions, in order
    span_start: list = field(default_factory=list)  # first logical position of each span S_k
    span_len: list = field(default_factory=list)    # |S_k| (0: no span after D_k)


def compose_layout(doc_len, doc_base_pos, doc_ids, prefix_len, query_len,
                   block_table, page_size=16, span_len=None) -> RequestLayout:
    """Assign logical positions in the order P, D_1, S_1, ..., D_m, S_m, Q and
    map them to slots.

    Walks the request from position 0: the prefix takes P positions, each
    document D_k takes the next n_k positions (its target offset) and its
    post-document inline span S_k the next |S_k| (``span_len[k]``, default 0),
    the query takes the final Tq positions.  A document cached at base
    position base_k therefore moves by delta_k = offset_k - base_k.  The
    inline tokens (prefix, spans, query, in this order) keep their own
    positions.  Logical position t lives in physical slot
    block_table[t // page_size] * page_size + t % page_size.
    """
    if span_len is None:
        span_len = [0] * len(doc_ids)
    if len(span_len) != len(doc_ids):
        raise ValueError("one span length per document")
    pos = int(prefix_len)
    offsets, deltas, span_start = [], [], []
    for d, s in zip(doc_ids, span_len):
        n = int(doc_len[d])
        if n <= 0:
            raise ValueError("document length must be positive")
        if int(s) < 0:
            raise ValueError("span length must not be negative")
        offsets.append(pos)
        deltas.append(pos - int(doc_base_pos[d]))
        pos += n
        span_start.append(pos)
        pos += int(s)
    query_start = pos
    ctx = pos + int(query_len)
    n_pages = -(-ctx // page_size)
    if n_pages > len(block_table):
        raise ValueError("block table shorter than the request")
    slots = np.empty(ctx, dtype=np.int64)
    for t in range(ctx):
        slots[t] = int(block_table[t // page_size]) * page_size + t % page_size
    inline_pos = np.concatenate(
        [np.arange(prefix_len)] + [np.arange(a, a + int(s)) for a, s in zip(span_start, span_len)]
        + [np.arange(query_start, ctx)]).astype(np.int64)
    return RequestLayout(int(prefix_len), list(doc_ids), offsets, deltas, query_start,
                         int(query_len), ctx, slots, inline_pos, span_start,
                         [int(s) for s in span_len])


# --------------------------------------------------------------------------
# Stitching: the dense logical context and its paged image
# --------------------------------------------------------------------------
def relocate_docs(layout: RequestLayout, k_docs, v_docs, doc_base_pos, theta, style=HALF):
    """Re-rotate each document's keys from its base to its target positions.

    ``k_docs[i]`` / ``v_docs[i]`` hold document layout.doc_ids[i] as compiled
    in isolation, shape [n_i, Hkv, d].  Token j of doc k sits at base position
    base_k + j and moves to offset_k + j (Eq. 3).  Returns the keys and values
    of all documents in order (concatenated), float64.
    """
    ks, vs = [], []
    for i, d in enumerate(layout.doc_ids):
        n = k_docs[i].shape[0]
        a = doc_base_pos[d] + np.arange(n)
        b = layout.doc_offset[i] + np.arange(n)
        ks.append(rerotate_key(k_docs[i], a[:, None], b[:, None], theta, style))
        vs.append(np.asarray(v_docs[i], dtype=np.float64))  # values are copied, not rotated
    if not ks:
        return None, None
    return np.concatenate(ks, 0), np.concatenate(vs, 0)


def dense_context(layout: RequestLayout, k_docs, v_docs, doc_base_pos,
                  k_inline, v_inline, theta, style=HALF, storage=None):
    """Keys/values of the whole request indexed by logical position.

    Inline tokens (prefix, spans, query, ``k_inline`` [P+S+Tq, Hkv, d]
    un-rotated) get RoPE at their own logical positions and are placed
    there; documents are relocated with Eq. 3 and placed at their offsets.
    Every position is filled exactly once.  Returns (K, V) of shape
    [ctx, Hkv, d].  storage="bf16" rounds the rotated keys to bf16, as a bf16
    cache holds them (values already are).
    """
    k_inline = np.asarray(k_inline, np.float64)
    ctx, (_, H, d) = layout.ctx_len, k_inline.shape
    K, V = np.zeros((ctx, H, d)), np.zeros((ctx, H, d))
    filled = np.zeros(ctx, dtype=np.int64)
    ip = layout.inline_pos
    K[ip] = rotary(k_inline, ip[:, None], theta, style)
    V[ip] = np.asarray(v_inline, np.float64)
    filled[ip] += 1
    kd, vd = relocate_docs(layout, k_docs, v_docs, doc_base_pos, theta, style)
    at = 0
    for i, off in enumerate(layout.doc_offset):
        n = k_docs[i].shape[0]
        K[off:off + n], V[off:off + n] = kd[at:at + n], vd[at:at + n]
        filled[off:off + n] += 1
        at += n
    assert (filled == 1).all(), "every logical position holds exactly one token"
    return _store(K, storage), V


def scatter_to_pages(layout: RequestLayout, K, V, k_cache, v_cache, page_size=16):
    """Write the logical sequence into a paged cache [pages, Hkv, page, d].

    This is the second route the tests use: the GPU's cache is compared after
    being read back through the same slot map.
    """
    for t in range(layout.ctx_len):
        page, off = divmod(int(layout.slot_mapping[t]), page_size)
        k_cache[page, :, off, :] = K[t]
        v_cache[page, :, off, :] = V[t]


def gather_from_pages(slot_mapping, k_cache, v_cache, page_size=16):
    """Read a paged cache [pages, Hkv, page, d] back in logical order."""
    pages = np.asarray(slot_mapping) // page_size
    offs = np.asarray(slot_mapping) % page_size
    return k_cache[pages, :, offs, :], v_cache[pages, :, offs, :]


# --------------------------------------------------------------------------
# Reader attention (unchanged decoder): GQA softmax under the frontier mask
# --------------------------------------------------------------------------
def attention(q, q_pos, K, V, k_pos=None, scale=None, return_lse=False):
    """Softmax attention of queries over logical keys under the frontier mask.

    q:  [T, Hq, d] rotated queries at logical positions q_pos [T]
    K, V: [S, Hkv, d] keys/values at logical positions k_pos [S] (default 0..S-1)
    Query head h reads kv head h // (Hq / Hkv).  Key s is visible to query t
    iff k_pos[s] <= q_pos[t].  Scores q.k * scale (scale = 1/sqrt(d)); the
    softmax subtracts the row maximum, exponentiates, normalises; the output
    is the probability-weighted sum of values.  float64 throughout.
    Returns O [T, Hq, d] (and the natural-log LSE [T, Hq] of the scaled scores).
    """
    q = np.asarray(q, np.float64)
    K = np.asarray(K, np.float64)
    V = np.asarray(V, np.float64)
    T, Hq, d = q.shape
    S, Hkv, _ = K.shape
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    k_pos = np.arange(S) if k_pos is None else np.asarray(k_pos)
    visible = k_pos[None, :] <= np.asarray(q_pos)[:, None]  # [T, S]
    out = np.zeros((T, Hq, d))
    lse = np.zeros((T, Hq))
    for h in range(Hq):
        g = h // G
        s = (q[:, h, :] @ K[:, g, :].T) * scale            # [T, S]
        s = np.where(visible, s, -np.inf)
        m = s.max(axis=1, keepdims=True)
        p = np.exp(s - m)
        z = p.sum(axis=1, keepdims=True)
        out[:, h, :] = (p / z) @ V[:, g, :]
        lse[:, h] = (m + np.log(z))[:, 0]
    return (out, lse) if return_lse else out


# --------------------------------------------------------------------------
# Whole path for one request and one layer
# --------------------------------------------------------------------------
def cache_hit_prefill(layout: RequestLayout, k_docs, v_docs, doc_base_pos,
                      q_inline, k_inline, v_inline, theta, style=HALF, return_lse=False,
                      storage=None):
    """Cache hit: relocate the docs, RoPE the inline tokens, attend.

    ``q_inline`` [T, Hq, d], ``k_inline`` / ``v_inline`` [T, Hkv, d] are the
    un-rotated projections of the T inline tokens (prefix, spans, query).
    Returns the attention output of every inline token, plus the dense (K, V)
    context the attention read.  storage="bf16": rotated keys and queries are
    rounded to bf16 before the (float64) attention.
    """
    K, V = dense_context(layout, k_docs, v_docs, doc_base_pos, k_inline, v_inline, theta, style,
                         storage)
    q_rot = _store(rotary(q_inline, layout.inline_pos[:, None], theta, style), storage)
    res = attention(q_rot, layout.inline_pos, K, V, return_lse=return_lse)
    return res, K, V


def decode_step(K, V, q_new, k_new, v_new, pos, theta, style=HALF, return_lse=False,
                storage=None):
    """One autoregressive step over a completed cache (ordinary decoding).

    The new token at logical position ``pos`` (== len(K)) is appended with its
    key rotated at ``pos``; its query, rotated at ``pos``, attends to every key
    0..pos.  Returns (output [Hq, d], K', V').
    """
    assert pos == K.shape[0]
    k_rot = _store(rotary(k_new, pos, theta, style), storage)
    K2 = np.concatenate([K, k_rot[None]], 0)
    V2 = np.concatenate([V, np.asarray(v_new, np.float64)[None]], 0)
    q_rot = _store(rotary(q_new, pos, theta, style), storage)
    res = attention(q_rot[None], np.array([pos]), K2, V2, return_lse=return_lse)
    if return_lse:
        return (res[0][0], res[1][0]), K2, V2
    return res[0], K2, V2


# --------------------------------------------------------------------------
# Attention-deviation diagnostic ("Motivating Analysis")
# --------------------------------------------------------------------------
def attention_probabilities(q, q_pos, K, k_pos=None, scale=None):
    """Post-softmax attention probabilities [T, Hq, S] of rotated queries q
    [T, Hq, d] at positions q_pos over keys K [S, Hkv, d] at k_pos (default
    0..S-1), frontier mask and GQA as in ``attention``; masked keys get 0."""
    q = np.asarray(q, np.float64)
    K = np.asarray(K, np.float64)
    T, Hq, d = q.shape
    S, Hkv, _ = K.shape
    G = Hq // Hkv
    scale = 1.0 / math.sqrt(d) if scale is None else scale
    k_pos = np.arange(S) if k_pos is None else np.asarray(k_pos)
    visible = k_pos[None, :] <= np.asarray(q_pos)[:, None]
    out = np.zeros((T, Hq, S))
    for h in range(Hq):
        s = (q[:, h, :] @ K[:, h // G, :].T) * scale
        s = np.where(visible, s, -np.inf)
        p = np.exp(s - s.max(axis=1, keepdims=True))
        out[:, h, :] = p / p.sum(axis=1, keepdims=True)
    return out


def block_region_bounds(n, edges):
    """Token index bounds of the normalized regions of a block of n tokens:
    region i holds the tokens j with edges[i] <= j / n < edges[i+1], i.e.
    ceil(edges[i] * n) <= j < ceil(edges[i+1] * n) (products in double
    precision)."""
    return [int(math.ceil(float(e) * n)) for e in edges]


def attention_deviation(q, q_pos, K_a, K_b, layout: RequestLayout, doc_lens, edges=(0.0, 0.1, 0.9)):
    """D_r(A, B) of the paper's diagnostic: the mean absolute deviation between
    the post-softmax attention probabilities of two configurations A and B
    (the same rotated queries over two key sets of one request, e.g. a
    relocated cache and one built another way) within normalized block
    region r.  Key t of the k-th block (document) lies at normalized
    position (t - offset_k) / n_k; region i is [edges[i], edges[i+1]) (the
    paper's pre = [0, 0.1), int = [0.1, 0.9)).

    Returns (sums, counts) per region: the sum over query rows, query heads
    and block keys in the region of |p_A - p_B|, and the number of terms; the
    deviation is sums / counts.
    """
    pa = attention_probabilities(q, q_pos, K_a)
    pb = attention_probabilities(q, q_pos, K_b)
    diff = np.abs(pa - pb)                      # [T, Hq, S]
    R = len(edges) - 1
    sums, counts = np.zeros(R), np.zeros(R, dtype=np.int64)
    T, Hq = diff.shape[:2]
    for off, n in zip(layout.doc_offset, doc_lens):
        b = block_region_bounds(n, edges)
        for i in range(R):
            lo, hi = off + b[i], off + max(b[i], b[i + 1])
            sums[i] += diff[:, :, lo:hi].sum()
            counts[i] += T * Hq * (hi - lo)
    return sums, counts
