"""Seeded synthetic inputs shaped like multi-document retrieval requests.

This module draws random numbers and sizes buffers; it holds none of the
method's arithmetic (no positions, rotations, slots or attention).  Both the
CUDA path and the CPU oracle receive the tensors made here.

Recipe (per workload): document K/V compiled at a base position (0 for the
five benchmark workloads; a per-document draw for parity cases that move
documents backwards as well as forwards; the paper's Writer is out of scope,
so the cached values are N(0,1) bf16 draws), a pool
of documents stored token-major ``[L][pool_tokens][Hkv][d]``, per-request
document choices in random order, an uncached inline prefix, a query chunk and
(optionally) decode tokens.  Physical pages are a seeded random permutation so
the stitched cache is genuinely scattered.  Values use seed 0, selections and
page permutations seed 1.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional

import numpy as np
import torch

PAGE = 16


@dataclass(frozen=True)
class WorkloadSpec:
    name: str
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    rope_base: float
    batch: int
    pool_docs: int
    docs_per_request: int
    doc_len: tuple            # (lo, hi) inclusive; lo == hi for fixed lengths
    prefix_len: tuple         # (lo, hi) inclusive
    query_len: int
    decode_steps: int = 0
    fixed_order: Optional[tuple] = None   # explicit doc order for every request
    shared_all_docs: bool = False         # every request uses the whole pool
    page_size: int = PAGE
    span_len: tuple = (0, 0)              # (lo, hi) inclusive: inline span S_k after each doc
    base_pos: tuple = (0, 0)              # (lo, hi) inclusive: compiled base position per pool doc
    description: str = ""


# The five workloads: sizes and structure of the paper's cache-hit requests
# (short records, multi-document QA, long-context retrieval), all synthetic.
WORKLOADS = {
    "tiny": WorkloadSpec(
        "tiny", 1, 4, 1, 64, 1e4, 1, 2, 2, (64, 64), (16, 16), 16,
        fixed_order=(0, 1),
        description="1 layer, 2 docs x 64 tokens relocated behind a 16-token prefix, "
                    "16 query tokens, Hq=4 Hkv=1 d=64, RoPE base 1e4"),
    "llama8b_1layer": WorkloadSpec(
        "llama8b_1layer", 1, 32, 8, 128, 5e5, 1, 32, 8, (512, 512), (64, 64), 128,
        description="one Llama-3-8B-shaped layer (32/8/128, base 5e5): 8 of 32 docs x 512 "
                    "tokens in random order, 64-token prefix, 128-token query chunk"),
    "llama8b_32layer_b8": WorkloadSpec(
        "llama8b_32layer_b8", 32, 32, 8, 128, 5e5, 8, 64, 16, (1024, 1024), (32, 128), 256,
        description="32 layers, batch 8, each request 16 of a shared 64-doc pool x 1024 "
                    "tokens, prefixes U{32..128}, 256-token query chunk"),
    "decode_28layer_b16": WorkloadSpec(
        "decode_28layer_b16", 28, 28, 4, 128, 1e6, 16, 64, 32, (1024, 1024), (64, 64), 128,
        decode_steps=128,
        description="28 layers (28/4/128, base 1e6), batch 16, 32 docs x 1024 tokens per "
                    "request from a 64-doc pool, 128-token query prefill then 128 decode steps"),
    "stress_128k_b4": WorkloadSpec(
        "stress_128k_b4", 32, 32, 8, 128, 5e5, 4, 128, 128, (128, 2048), (64, 64), 512,
        shared_all_docs=True,
        description="32 layers, batch 4 requests of ~139k tokens: all 128 docs of a pool with "
                    "lengths U{128..2048}, each request in its own shuffled order, "
                    "512-token query chunk"),
    # The 32-layer batch-8 workload with a request-time inline span S_k of
    # 16-64 tokens after every document (canonical order P, D_1, S_1, ...,
    # D_m, S_m, Q): ~640 more inline tokens per request.
    "llama8b_32layer_b8_spans": WorkloadSpec(
        "llama8b_32layer_b8_spans", 32, 32, 8, 128, 5e5, 8, 64, 16, (1024, 1024), (32, 128), 256,
        span_len=(16, 64),
        description="llama8b_32layer_b8 with an inline span of U{16..64} tokens after each "
                    "document"),
    # Profiling-size slices of the full workloads (same per-layer shapes, fewer
    # layers / steps), so that one profiled launch moves more than L2 holds
    # while the process stays at a few GB of device memory.
    "llama8b_2layer_b8": WorkloadSpec(
        "llama8b_2layer_b8", 2, 32, 8, 128, 5e5, 8, 64, 16, (1024, 1024), (32, 128), 256,
        description="2 layers of llama8b_32layer_b8 (profiling slice)"),
    "decode_1layer_b16": WorkloadSpec(
        "decode_1layer_b16", 1, 28, 4, 128, 1e6, 16, 64, 32, (1024, 1024), (64, 64), 128,
        decode_steps=1,
        description="1 layer of decode_28layer_b16 with one decode step (profiling slice)"),
    "stress_1layer_b4": WorkloadSpec(
        "stress_1layer_b4", 1, 32, 8, 128, 5e5, 4, 128, 128, (128, 2048), (64, 64), 512,
        shared_all_docs=True,
        description="1 layer of stress_128k_b4 (profiling slice)"),
}


@dataclass
class Workload:
    spec: WorkloadSpec
    # document pool
    doc_len: torch.Tensor          # [n_pool] int32
    doc_base_pos: torch.Tensor     # [n_pool] int32 (0: compiled in isolation)
    doc_token_start: torch.Tensor  # [n_pool] int64 row of the doc's first token
    k_pool: torch.Tensor           # [L][pool_tokens][Hkv][d] bf16
    v_pool: torch.Tensor
    # requests
    req_doc_ids: torch.Tensor      # [B][max_docs] int32 (-1 padded)
    req_num_docs: torch.Tensor     # [B] int32
    prefix_len: torch.Tensor       # [B] int32
    query_len: torch.Tensor        # [B] int32
    block_table: torch.Tensor      # [B][max_pages] int32 (-1 padded)
    num_pages: int
    max_ctx: int                   # upper bound on prompt context per request
    # inline projections (un-rotated), prefix tokens then query tokens
    q_inline: torch.Tensor         # [L][B][Tin_max][Hq][d] bf16
    k_inline: torch.Tensor         # [L][B][Tin_max][Hkv][d] bf16
    v_inline: torch.Tensor
    inline_len: torch.Tensor       # [B] int32 (prefix + span + query tokens)
    # decode tokens
    q_dec: Optional[torch.Tensor] = None   # [steps][L][B][Hq][d]
    k_dec: Optional[torch.Tensor] = None   # [steps][L][B][Hkv][d]
    v_dec: Optional[torch.Tensor] = None
    meta: dict = field(default_factory=dict)
    span_len: Optional[torch.Tensor] = None   # [B][max_docs] int32 (0-padded), None: no spans

    @property
    def tin_max(self) -> int:
        return self.q_inline.shape[2]


def _randn_bf16(shape, gen, device):
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    # Chunked along the leading dim to bound the fp32 temporary.
    flat = out.view(shape[0], -1) if len(shape) > 1 else out.view(1, -1)
    for i in range(flat.shape[0]):
        flat[i].copy_(torch.randn(flat.shape[1], generator=gen, device=device,
                                  dtype=torch.float32))
    return out


@dataclass
class Structure:
    """The selections of a workload, without any tensor: pool document
    lengths, rows and base positions, each request's documents, prefix and
    spans, and its block table.  Cheap at every size (the bench's CPU arm
    reads its shape from here)."""
    lens: np.ndarray          # [n_pool] int64
    starts: np.ndarray        # [n_pool] int64 first pool row of each document
    bases: np.ndarray         # [n_pool] int64 compiled base position
    docs: list                # per request: pool ids in request order
    prefixes: list            # per request: prefix length
    spans: list               # per request: span length after each document
    block_table: np.ndarray   # [B][max_pages] int32 (-1 padded)
    num_pages: int
    need: list                # per request: positions incl. decode tokens
    tin: list                 # per request: inline tokens (prefix + spans + query)

    @property
    def pool_tokens(self) -> int:
        return int(self.lens.sum())


def draw_structure(spec, select_seed=1) -> Structure:
    """Draw the selections of a workload with the selection seed."""
    if isinstance(spec, str):
        spec = WORKLOADS[spec]
    rng = np.random.default_rng(select_seed)
    B = spec.batch
    lo, hi = spec.doc_len
    lens = np.full(spec.pool_docs, lo, np.int64) if lo == hi else \
        rng.integers(lo, hi + 1, size=spec.pool_docs)
    starts = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int64)

    docs = []
    for b in range(B):
        if spec.fixed_order is not None:
            docs.append(list(spec.fixed_order))
        elif spec.shared_all_docs:
            docs.append(list(rng.permutation(spec.pool_docs)))
        else:
            docs.append(list(rng.choice(spec.pool_docs, spec.docs_per_request, replace=False)))
    plo, phi = spec.prefix_len
    prefixes = [int(plo) if plo == phi else int(rng.integers(plo, phi + 1)) for _ in range(B)]
    # post-document inline spans S_k (drawn only when the spec asks for them,
    # so the other workloads keep their draws)
    slo, shi = spec.span_len
    spans = [[0] * len(docs[b]) for b in range(B)]
    if shi > 0:
        spans = [[int(x) for x in rng.integers(slo, shi + 1, size=len(docs[b]))] for b in range(B)]

    # Page budget per request: prompt plus decode tokens.
    need = [prefixes[b] + int(lens[docs[b]].sum()) + sum(spans[b]) + spec.query_len
            + spec.decode_steps for b in range(B)]
    pages_per_req = [-(-n // spec.page_size) for n in need]
    num_pages = int(sum(pages_per_req))
    perm = rng.permutation(num_pages).astype(np.int32)
    max_pages = max(pages_per_req)
    bt = np.full((B, max_pages), -1, np.int32)
    o = 0
    for b in range(B):
        bt[b, :pages_per_req[b]] = perm[o:o + pages_per_req[b]]
        o += pages_per_req[b]
    # compiled base positions, drawn last and only when asked for (the other
    # workloads keep every draw above)
    blo, bhi = spec.base_pos
    bases = np.zeros(spec.pool_docs, np.int64)
    if (blo, bhi) != (0, 0):
        bases = rng.integers(blo, bhi + 1, size=spec.pool_docs).astype(np.int64)
    tin = [prefixes[b] + sum(spans[b]) + spec.query_len for b in range(B)]
    return Structure(lens, starts, bases, docs, prefixes, spans, bt, num_pages, need, tin)


def generate(spec, device="cpu", gen_device=None, value_seed=0, select_seed=1) -> Workload:
    """Materialise a workload.  ``gen_device`` selects the random generator
    ('cpu' for sizes the oracle handles, 'cuda' for the full-size ones);
    tensors end up on ``device``."""
    if isinstance(spec, str):
        spec = WORKLOADS[spec]
    gen_device = gen_device or device
    st = draw_structure(spec, select_seed)
    L, Hq, Hkv, d, B = spec.layers, spec.q_heads, spec.kv_heads, spec.head_dim, spec.batch
    docs, spans, lens = st.docs, st.spans, st.lens
    pool_tokens = st.pool_tokens
    max_docs = max(len(x) for x in docs)
    ids = np.full((B, max_docs), -1, np.int32)
    for b in range(B):
        ids[b, :len(docs[b])] = docs[b]

    gen = torch.Generator(device=gen_device)
    gen.manual_seed(value_seed)
    k_pool = _randn_bf16((L, pool_tokens, Hkv, d), gen, gen_device)
    v_pool = _randn_bf16((L, pool_tokens, Hkv, d), gen, gen_device)
    tin_max = max(st.tin)
    q_in = _randn_bf16((L, B, tin_max, Hq, d), gen, gen_device)
    k_in = _randn_bf16((L, B, tin_max, Hkv, d), gen, gen_device)
    v_in = _randn_bf16((L, B, tin_max, Hkv, d), gen, gen_device)
    qd = kd = vd = None
    if spec.decode_steps:
        s = spec.decode_steps
        qd = _randn_bf16((s, L, B, Hq, d), gen, gen_device)
        kd = _randn_bf16((s, L, B, Hkv, d), gen, gen_device)
        vd = _randn_bf16((s, L, B, Hkv, d), gen, gen_device)

    def i32(x):
        return torch.as_tensor(np.asarray(x), dtype=torch.int32).to(device)

    mv = lambda t: None if t is None else t.to(device)  # noqa: E731
    return Workload(
        spec=spec,
        doc_len=i32(lens), doc_base_pos=i32(st.bases),
        doc_token_start=torch.as_tensor(st.starts, dtype=torch.int64).to(device),
        k_pool=mv(k_pool), v_pool=mv(v_pool),
        req_doc_ids=i32(ids), req_num_docs=i32([len(x) for x in docs]),
        prefix_len=i32(st.prefixes), query_len=i32([spec.query_len] * B),
        block_table=i32(st.block_table), num_pages=st.num_pages, max_ctx=max(st.need),
        q_inline=mv(q_in), k_inline=mv(k_in), v_inline=mv(v_in), inline_len=i32(st.tin),
        q_dec=mv(qd), k_dec=mv(kd), v_dec=mv(vd),
        meta={"docs": docs, "prefix": st.prefixes, "pool_tokens": pool_tokens, "spans": spans},
        span_len=i32([x + [0] * (max_docs - len(x)) for x in spans])
        if spec.span_len[1] > 0 else None,
    )


def custom_spec(**kw) -> WorkloadSpec:
    """A small workload for tests (defaults: tiny shape)."""
    base = dict(name="custom", layers=1, q_heads=4, kv_heads=1, head_dim=64, rope_base=1e4,
                batch=1, pool_docs=2, docs_per_request=2, doc_len=(64, 64),
                prefix_len=(16, 16), query_len=16)
    base.update(kw)
    return WorkloadSpec(**base)


def bf16_round_trip_ok(x: torch.Tensor) -> bool:
    """True when every element is finite (sanity check on generated inputs)."""
    return bool(torch.isfinite(x.float()).all())


def pages_for(tokens: int, page_size: int = PAGE) -> int:
    return int(math.ceil(tokens / page_size))
