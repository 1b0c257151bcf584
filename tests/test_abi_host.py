"""Host-side checks of the C ABI (no GPU needed): the library builds and loads,
exports every function include/pic.h declares, and the calls that never reach
the device (version, workspace sizes, argument validation) behave."""
import ctypes
import os
import re

import pytest

import paper_2607_28069_gb300 as pic

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pic.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(pic.lib_path()):
        from paper_2607_28069_gb300.build import build
        build()
    return pic.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(pic_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_binding_symbols():
    assert declared_functions() == sorted(pic.EXPORTED_SYMBOLS)


def test_library_exports_every_declared_symbol(lib):
    missing = [s for s in declared_functions() if not hasattr(lib, s)]
    assert not missing, missing


def test_version(lib):
    assert pic.pic_abi_version() == 4


def _geom(**kw):
    g = dict(num_layers=2, num_q_heads=32, num_kv_heads=8, head_dim=128, rope_base=5e5)
    g.update(kw)
    return pic.Geometry(**g)


def test_workspace_sizes_are_host_arithmetic(lib):
    g = _geom()
    # packed Q: B * Hkv * ceil(Tin*G/128)*128 rows of d bf16
    ws1 = pic.pic_prefill_workspace_size(g, 1, 192, 4288, 1)
    assert ws1 == 1 * 8 * 768 * 128 * 2
    # rotate-on-load adds a 16-byte source per page of max_ctx and d/2 cos/sin
    # pairs per listed document
    wf = pic.pic_prefill_fused_workspace_size(g, 1, 192, 4288, 8, 1)
    assert wf == ws1 + ((268 * 16 + 255) // 256) * 256 + 8 * 64 * 8
    ws3 = pic.pic_prefill_workspace_size(g, 1, 192, 4288, 3)
    assert ws3 > ws1
    assert pic.pic_decode_workspace_size(g, 16, 33000, 1) == ((16 * 32 * 128 * 2 + 255) // 256) * 256
    assert pic.pic_decode_workspace_size(_geom(num_kv_heads=0), 1, 10, 1) == 0
    # one Llama-3-8B layer, 192 inline tokens over ~4.3k keys: 48 query tiles in
    # 24 two-tile CTAs; six key splits fill the GPU in a single wave
    assert pic.pic_prefill_num_splits(g, 1, 192, 4288, 0) == 6
    assert pic.pic_prefill_num_splits(g, 1, 192, 4288, 5) == 5
    assert pic.pic_decode_num_splits(g, 16, 33000, 7) == 7
    assert 1 <= pic.pic_decode_num_splits(g, 16, 33000, 0) <= 64


def _call_compose_with(geom):
    g = geom._c()
    null = ctypes.c_void_p(0)
    return pic.load().pic_compose(ctypes.byref(g), 1, 1, 1, null, null, null, null, null, null,
                                  null, null, null, 1, 1, 16, 16, null, null, null, null, null,
                                  null, null)


def test_invalid_geometry_rejected_before_launch(lib):
    assert _call_compose_with(_geom(head_dim=96)) == 2          # PIC_ERR_UNSUPPORTED
    assert b"head_dim" in pic.load().pic_last_error()
    assert _call_compose_with(_geom(num_kv_heads=5)) == 1       # Hq % Hkv != 0
    assert _call_compose_with(_geom(page_size=32)) == 2
    assert _call_compose_with(_geom(rope_base=1.0)) == 1
    assert _call_compose_with(_geom(rope_style=7)) == 1
    # valid geometry but NULL tensors: still rejected on the host
    assert _call_compose_with(_geom()) == 1
    assert b"NULL" in pic.load().pic_last_error()


def test_inv_freq_override_validated(lib):
    bad = _geom(head_dim=64, inv_freq=[1.0] * 31 + [-1.0])
    assert _call_compose_with(bad) == 1
    assert b"inv_freq" in pic.load().pic_last_error()


def test_binding_rejects_cpu_tensors():
    import torch
    with pytest.raises(ValueError):
        pic._ptr(torch.zeros(4, dtype=torch.int32), torch.int32, "x")


def test_product_path_does_not_import_the_oracle():
    pkg = os.path.join(ROOT, "paper_2607_28069_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in src and "from oracle" not in src, f


def _call_deviation_with(geom, edges, n_regions, layer=0, tensors=True):
    g = geom._c()
    null = ctypes.c_void_p(0)
    fake = ctypes.c_void_p(256) if tensors else null   # never dereferenced: rejected first
    arr = (ctypes.c_double * len(edges))(*edges)
    return pic.load().pic_attention_deviation(
        ctypes.byref(g), layer, 1, 16, 2, 64, 8,
        fake, fake, fake, 4,                      # inline_pos, inline_len, query_len, max_query_len
        fake, fake, fake, fake,                   # req_doc_ids, doc_len, doc_offset, slots
        fake, fake, fake, fake,                   # k_cache_a, k_cache_b, lse_a, lse_b
        ctypes.cast(arr, ctypes.c_void_p), n_regions, fake, 1 << 20, fake, fake, null)


def test_attention_deviation_arguments_checked_on_the_host(lib):
    g = _geom()
    assert _call_deviation_with(g, [0.0, 0.1, 0.9], 0) == 1        # no region
    assert _call_deviation_with(g, [0.0] * 10, 9) == 1              # more than 8 regions
    assert _call_deviation_with(g, [0.0, 0.9, 0.1], 2) == 1         # edges not ascending
    assert b"edges" in pic.load().pic_last_error()
    assert _call_deviation_with(g, [0.0, 1.5], 1) == 1              # outside [0, 1]
    assert _call_deviation_with(g, [0.0, 0.1, 0.9], 2, layer=2) == 1  # layer outside the model
    assert _call_deviation_with(g, [0.0, 0.1, 0.9], 2, tensors=False) == 1
    assert b"NULL" in pic.load().pic_last_error()


def test_geometry_binding_carries_the_per_layer_table_pointer():
    import torch
    g = _geom()
    assert g._c().layer_inv_freq is None
    with pytest.raises(ValueError):   # wrong shape is refused before any call
        pic.Geometry(2, 32, 8, 128, 5e5, layer_inv_freq=torch.zeros((3, 64),
                                                                     dtype=torch.float64))._c()


def test_compose_span_input_is_optional_in_the_binding():
    import inspect
    for fn in (pic.pic_compose, pic.pic_link):
        assert inspect.signature(fn).parameters["span_len"].default is None


def test_copy_binding_refuses_pageable_and_mismatched_tensors():
    import torch
    a = torch.zeros(64, dtype=torch.uint8)           # pageable host memory
    with pytest.raises(ValueError):
        pic.pic_copy_async(a, torch.zeros(64, dtype=torch.uint8))
    with pytest.raises(ValueError):
        pic.pic_copy_async(a[::2], a[1::2])            # not contiguous


def test_launch_probe_rejects_bad_shapes_before_any_launch(lib):
    import ctypes as C
    g = (C.c_int32 * 3)(1, 1, 1)
    b = (C.c_int32 * 1)(32)
    m = (C.c_int32 * 1)(0)
    assert pic.load().pic_launch_probe(0, g, b, m, None) == 1      # n must be positive
    assert pic.load().pic_launch_probe(1, None, b, m, None) == 1   # arrays required


def test_wait_probe_rejects_its_limit_on_the_host(lib):
    assert pic.load().pic_wait_probe(0, 10, None) == 1            # below 1 us
    assert pic.load().pic_wait_probe(1, 10 ** 11, None) == 1      # above 10 s
    assert b"limit_ns" in pic.load().pic_last_error()
