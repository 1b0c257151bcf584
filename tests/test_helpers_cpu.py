"""The comparison bars the GPU tests use, checked on the CPU against what
bfloat16 rounding fixes (no GPU, no oracle arithmetic)."""
import numpy as np
import torch

from tests.helpers import attn_close, half_ulp_bf16, kv_tolerance_ok


def test_half_ulp_of_bfloat16_by_binade():
    # 8 significant bits: the spacing in [2^e, 2^(e+1)) is 2^(e-7)
    x = np.array([1.0, 1.5, 1.99, 2.0, 3.9, 0.75, 0.5, 2.0 ** -20, -6.0])
    want = np.array([2.0 ** -8, 2.0 ** -8, 2.0 ** -8, 2.0 ** -7, 2.0 ** -7, 2.0 ** -9,
                     2.0 ** -9, 2.0 ** -28, 2.0 ** -6])
    assert np.array_equal(half_ulp_bf16(x), want)


def test_half_ulp_bounds_torch_bfloat16_rounding():
    """Rounding to bf16 (torch's conversion, round to nearest even) moves a
    value by at most half an ulp of the rounded value, the allowance the
    attention bar adds to 1e-2."""
    g = torch.Generator().manual_seed(5)
    x = (torch.randn(200_000, generator=g, dtype=torch.float32) * 8.0)
    r = x.to(torch.bfloat16).to(torch.float64)
    x = x.to(torch.float64)
    err = (r - x).abs().numpy()
    assert (err <= half_ulp_bf16(np.maximum(np.abs(r.numpy()), np.abs(x.numpy())))).all()
    # and the bound is attained up to rounding: some element sits near it
    assert (err / half_ulp_bf16(np.abs(r.numpy()))).max() > 0.99


def test_attention_bar_admits_bf16_storage_and_rejects_1e2_more():
    g = np.random.default_rng(0)
    ref = g.normal(size=(64, 8, 128)) * 3.0
    stored = torch.tensor(ref).to(torch.bfloat16).double().numpy()
    ok, ratio, row = attn_close(stored, ref)
    assert ok and ratio <= 1.0 and row < 1e-2
    bad = stored.copy()
    bad[3, 2, 7] += 1.2e-2 + 2.0 ** -6          # beyond 1e-2 plus half an ulp below 8
    ok, ratio, _ = attn_close(bad, ref)
    assert not ok and ratio > 1.0


def test_attention_bar_is_the_plain_1e2_for_small_outputs():
    ref = np.full((4, 2, 16), 0.01)
    ok, _, _ = attn_close(ref + 0.0099, ref, row_rel=10.0)
    assert ok
    ok, _, _ = attn_close(ref + 0.0105, ref, row_rel=10.0)
    assert not ok


def test_key_bar_admits_bf16_rounding_of_exact_keys():
    g = np.random.default_rng(1)
    ref = g.normal(size=(300, 4, 128))
    stored = torch.tensor(ref).to(torch.bfloat16).double().numpy()
    ok, ratio = kv_tolerance_ok(stored, ref)
    assert ok and ratio < 1.0
