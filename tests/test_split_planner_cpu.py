"""Host-side split planning (no GPU): the inline positions the pipeline
derives on the host agree with the oracle's layout, and the planner returns
a count the kernels accept."""
import numpy as np
import pytest
import torch

import paper_2607_28069_gb300 as pic
from paper_2607_28069_gb300.pipeline import host_inline_positions
from paper_2607_28069_gb300.workloads import WORKLOADS, generate

from helpers import oracle_layout
from test_gpu_parity import SMALL


@pytest.mark.parametrize("name", ["tiny", "ragged_b3", "spans_b2", "boundary_blocks",
                                  "base_mixed", "no_docs"])
def test_host_inline_positions_match_the_oracle_layout(name):
    wl = generate(SMALL[name], device="cpu", gen_device="cpu")
    lens, pos = host_inline_positions(wl)
    for b in range(wl.spec.batch):
        ref = oracle_layout(wl, b).inline_pos
        assert int(lens[b]) == len(ref) == int(wl.inline_len[b])
        assert np.array_equal(pos[b, :len(ref)].numpy(), np.asarray(ref, dtype=np.int32))


def test_planner_returns_a_valid_split_count():
    spec = WORKLOADS["llama8b_32layer_b8"]
    g = pic.Geometry(1, spec.q_heads, spec.kv_heads, spec.head_dim, spec.rope_base)
    # query rows that see ~16.7k keys behind prefixes of 32..128 tokens
    B, tmax = 8, 128 + 256
    lens = torch.zeros(B, dtype=torch.int32)
    pos = torch.zeros((B, tmax), dtype=torch.int32)
    for b in range(B):
        p = 32 + 12 * b
        row = list(range(p)) + list(range(16384 + p, 16384 + p + 256))
        lens[b] = len(row)
        pos[b, :len(row)] = torch.tensor(row, dtype=torch.int32)
    s = pic.pic_prefill_plan_splits(g, 16384 + 128 + 256, lens, pos)
    assert 1 <= s <= 32
    # a single short request fills a fraction of the GPU: more splits than one
    one = pic.pic_prefill_plan_splits(g, 4096, torch.tensor([192], dtype=torch.int32),
                                      torch.arange(4096 - 192, 4096, dtype=torch.int32)[None])
    assert one > 1
    with pytest.raises(ValueError):
        pic.pic_prefill_plan_splits(g, 4096, lens, pos[0])
