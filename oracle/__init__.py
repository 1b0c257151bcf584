"""CPU oracle for the SemPIC cache-hit path (test infrastructure only).

Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline and
``--impl reference`` legs may import this package; the product path never does.
"""
from .pic_oracle import (  # noqa: F401
    HALF, INTERLEAVED, RequestLayout, attention, attention_deviation, attention_probabilities,
    block_region_bounds, cache_hit_prefill, compose_layout,
    decode_step, dense_context, gather_from_pages, relocate_docs, rerotate_key, round_bf16,
    rope_frequencies, rotary, scatter_to_pages,
)
