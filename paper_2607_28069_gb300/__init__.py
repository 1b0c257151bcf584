"""SemPIC cache-hit path on GB300: thin Python binding of libpic.so.

The functions below carry the names of the C entry points in include/pic.h
and only marshal arguments (device pointers of torch tensors, sizes, the
current CUDA stream).  Every step of the path runs in the CUDA kernels of
libpic.so; if the library is missing, the calls raise -- there is no CPU
fallback.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

__all__ = [
    "Geometry", "load", "lib_path", "pic_abi_version", "pic_compose", "pic_relocate",
    "pic_relocate_mapped", "pic_link",
    "pic_attention_deviation", "pic_copy_async", "pic_launch_probe", "pic_wait_probe",
    "pic_append_inline", "pic_attend_prefill", "pic_attend_prefill_fused",
    "pic_prefill_workspace_size", "pic_prefill_fused_workspace_size",
    "pic_prefill_num_splits", "pic_prefill_plan_splits", "pic_decode_num_splits",
    "pic_attend_decode_noalloc",
    "pic_attend_decode", "pic_decode_workspace_size", "pic_device_status", "PicError",
    "EXPORTED_SYMBOLS", "ROPE_HALF", "ROPE_INTERLEAVED",
]

_PKG = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_PKG, "libpic.so")
_lib = None

ROPE_HALF = 0
ROPE_INTERLEAVED = 1

# Every symbol include/pic.h declares.
EXPORTED_SYMBOLS = (
    "pic_abi_version", "pic_last_error", "pic_device_status", "pic_compose", "pic_relocate",
    "pic_relocate_mapped", "pic_link", "pic_attention_deviation", "pic_prefill_workspace_size",
    "pic_prefill_fused_workspace_size", "pic_prefill_num_splits", "pic_prefill_plan_splits",
    "pic_append_inline",
    "pic_attend_prefill", "pic_attend_prefill_fused", "pic_decode_workspace_size", "pic_decode_num_splits",
    "pic_attend_decode", "pic_attend_decode_noalloc", "pic_copy_async", "pic_launch_probe",
    "pic_wait_probe",
)

DEVICE_CODES = {
    0: "ok", 1: "bad doc id", 2: "bad doc length", 3: "bad request", 4: "context overflow",
    5: "block table short", 6: "bad page", 7: "bad position", 8: "timeout",
}


class PicError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"libpic status {status}: {msg}")
        self.status = status


class _Geom(ctypes.Structure):
    _fields_ = [
        ("num_layers", ctypes.c_int32), ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32), ("rope_style", ctypes.c_int32),
        ("rope_base", ctypes.c_double), ("inv_freq", ctypes.POINTER(ctypes.c_double)),
        ("layer_inv_freq", ctypes.c_void_p),
    ]


@dataclass
class Geometry:
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    rope_base: float
    page_size: int = 16
    rope_style: int = ROPE_HALF
    inv_freq: Optional[list] = None
    # device float64 [num_layers][head_dim / 2]: a rotary table per layer
    layer_inv_freq: Optional[torch.Tensor] = None

    def _c(self):
        g = _Geom(self.num_layers, self.num_q_heads, self.num_kv_heads, self.head_dim,
                  self.page_size, self.rope_style, float(self.rope_base), None, None)
        if self.inv_freq is not None:
            arr = (ctypes.c_double * len(self.inv_freq))(*[float(x) for x in self.inv_freq])
            g.inv_freq = ctypes.cast(arr, ctypes.POINTER(ctypes.c_double))
            g._keep = arr  # keep the array alive with the struct
        if self.layer_inv_freq is not None:
            t = self.layer_inv_freq
            if tuple(t.shape) != (self.num_layers, self.head_dim // 2):
                raise ValueError("layer_inv_freq must be [num_layers][head_dim / 2]")
            g.layer_inv_freq = _ptr(t, torch.float64, "layer_inv_freq")
        return g


def lib_path() -> str:
    return _LIB_PATH


def load():
    """Load libpic.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"{_LIB_PATH} is missing: run __graft_entry__.build() first")
    lib = ctypes.CDLL(_LIB_PATH)
    P, I32, I64, SZ, D = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_double
    G = ctypes.POINTER(_Geom)
    sig = {
        "pic_abi_version": (I32, []),
        "pic_last_error": (ctypes.c_char_p, []),
        "pic_device_status": (I32, [P, P, P]),
        "pic_copy_async": (I32, [P, P, SZ, P]),
        "pic_launch_probe": (I32, [I32, P, P, P, P]),
        "pic_wait_probe": (I32, [I32, I64, P]),
        "pic_compose": (I32, [G, I32, I32, I32, P, P, P, P, P, P, P, P, P, I32, I64, I32, I32,
                              P, P, P, P, P, P, P]),
        "pic_relocate": (I32, [G, I32, I32, I32, P, P, I64, P, P, P, P, P, P, P, I32, I64, P, P,
                               I32, I32, P]),
        "pic_relocate_mapped": (I32, [G, I32, I32, P, P, I64, P, P, P, I32, I64, P, P, I32, I32,
                                      P]),
        "pic_link": (I32, [G, I32, I32, I32, P, P, P, P, P, P, P, P, P, I32, I64, I32, I32, P, P, I64,
                           I32, I32, I32, P, P, P, P, P, P, P, P, P, P, P, P, P, SZ, P]),
        "pic_prefill_workspace_size": (SZ, [G, I32, I32, I32, I32]),
        "pic_prefill_fused_workspace_size": (SZ, [G, I32, I32, I32, I32, I32]),
        "pic_attention_deviation": (I32, [G, I32, I32, I32, I32, I32, I64, P, P, P, I32, P, P, P,
                                          P, P, P, P, P, P, I32, P, SZ, P, P, P]),
        "pic_append_inline": (I32, [G, I32, I32, I32, P, P, P, P, P, P, I32, I64, P, P, P, SZ,
                                    P]),
        "pic_attend_prefill": (I32, [G, I32, I32, I32, P, P, P, P, P, I32, P, I32, I64, P, P, P,
                                     P, I32, P, SZ, P]),
        "pic_attend_prefill_fused": (I32, [G, I32, I32, I32, P, P, P, P, P, I32, P, I32, I64, P,
                                           P, P, P, I64, I32, P, P, P, P, I32, P, SZ, P]),
        "pic_decode_workspace_size": (SZ, [G, I32, I32, I32]),
        "pic_attend_decode_noalloc": (I32, [G, I32, I32, P, P, P, P, I32, P, I32, I64, P, P, P, P,
                                            I32, I32, P]),
        "pic_prefill_num_splits": (I32, [G, I32, I32, I32, I32]),
        "pic_prefill_plan_splits": (I32, [G, I32, I32, I32, P, P]),
        "pic_decode_num_splits": (I32, [G, I32, I32, I32]),
        "pic_attend_decode": (I32, [G, I32, I32, P, P, P, P, I32, P, I32, I64, P, P, P, P, I32, I32,
                                    P, SZ, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    del D
    _lib = lib
    return lib


def _check(status: int, what: str):
    if status != 0:
        msg = _lib.pic_last_error().decode(errors="replace")
        raise PicError(status, f"{what}: {msg}")


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr_or_pinned(t: torch.Tensor, dtype, name: str):
    """Like _ptr, for an output that may also live in pinned host memory."""
    if not t.is_cuda and t.is_pinned():
        if t.dtype != dtype or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous {dtype} tensor")
        return ctypes.c_void_p(t.data_ptr())
    return _ptr(t, dtype, name)


def _ptr(t: Optional[torch.Tensor], dtype, name: str, allow_none=False):
    if t is None:
        if allow_none:
            return None
        raise ValueError(f"{name} is required")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


bf16, i32, i64, f32 = torch.bfloat16, torch.int32, torch.int64, torch.float32


def pic_abi_version() -> int:
    return load().pic_abi_version()


def pic_device_status(stream=None):
    """(code, detail) of the first device-side failure since the last read; clears it."""
    lib = load()
    code, detail = ctypes.c_int32(0), ctypes.c_int32(0)
    st = lib.pic_device_status(_stream(stream), ctypes.byref(code), ctypes.byref(detail))
    if st not in (0, 5):
        _check(st, "pic_device_status")
    return code.value, detail.value


def pic_copy_async(dst: torch.Tensor, src: torch.Tensor, stream=None):
    """Copy the bytes of src into dst (see include/pic.h): each a contiguous
    CUDA tensor of the current device or a pinned CPU tensor, of the same
    size in bytes.  The GPU's own loads and stores move them."""
    for t, name in ((dst, "dst"), (src, "src")):
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
        if not t.is_cuda and not t.is_pinned():
            raise ValueError(f"{name} must be a CUDA tensor or pinned host memory")
    nbytes = dst.numel() * dst.element_size()
    if src.numel() * src.element_size() != nbytes:
        raise ValueError("dst and src differ in size")
    st = load().pic_copy_async(ctypes.c_void_p(dst.data_ptr()), ctypes.c_void_p(src.data_ptr()),
                               nbytes, _stream(stream))
    _check(st, "pic_copy_async")


def pic_launch_probe(shapes, stream=None):
    """Launch empty programmatic-dependent kernels with the given shapes, a
    list of (grid (x, y, z), block threads, dynamic shared bytes)."""
    n = len(shapes)
    grid = (ctypes.c_int32 * (3 * n))(*[int(g) for s in shapes for g in s[0]])
    block = (ctypes.c_int32 * n)(*[int(s[1]) for s in shapes])
    smem = (ctypes.c_int32 * n)(*[int(s[2]) for s in shapes])
    st = load().pic_launch_probe(n, grid, block, smem, _stream(stream))
    _check(st, "pic_launch_probe")


def pic_wait_probe(arrive: bool, limit_ns: int, stream=None):
    """One bounded mbarrier wait of limit_ns on the device: completes when
    `arrive`, else runs out and records a timeout in the device status word
    (read it with pic_device_status)."""
    st = load().pic_wait_probe(1 if arrive else 0, int(limit_ns), _stream(stream))
    _check(st, "pic_wait_probe")


def pic_compose(geom: Geometry, doc_len, doc_base_pos, doc_token_start, req_doc_ids,
                req_num_docs, prefix_len, query_len, block_table, num_pages: int, max_ctx: int,
                max_inline: int, doc_offset, doc_delta, slot_mapping, tok_map, inline_pos,
                ctx_len, stream=None, span_len=None):
    """span_len: int32 [batch][max_docs] post-document inline span lengths, or None."""
    lib = load()
    g = geom._c()
    B, max_docs = req_doc_ids.shape
    st = lib.pic_compose(
        ctypes.byref(g), B, max_docs, doc_len.numel(), _ptr(doc_len, i32, "doc_len"),
        _ptr(doc_base_pos, i32, "doc_base_pos"), _ptr(doc_token_start, i64, "doc_token_start"),
        _ptr(req_doc_ids, i32, "req_doc_ids"), _ptr(req_num_docs, i32, "req_num_docs"),
        _ptr(span_len, i32, "span_len", allow_none=True),
        _ptr(prefix_len, i32, "prefix_len"), _ptr(query_len, i32, "query_len"),
        _ptr(block_table, i32, "block_table"), block_table.shape[1], num_pages, max_ctx,
        max_inline, _ptr(doc_offset, i32, "doc_offset"), _ptr(doc_delta, i32, "doc_delta"),
        _ptr(slot_mapping, i64, "slot_mapping"), _ptr(tok_map, i64, "tok_map"),
        _ptr(inline_pos, i32, "inline_pos"), _ptr(ctx_len, i32, "ctx_len"), _stream(stream))
    _check(st, "pic_compose")


def pic_relocate(geom: Geometry, k_pool, v_pool, doc_token_start, doc_len, doc_base_pos,
                 req_doc_ids, req_num_docs, doc_target, block_table, num_pages: int, k_cache,
                 v_cache, layer_begin: int, layer_end: int, stream=None):
    """Per-document relocation: request b's k-th listed document moves from
    its base position to doc_target[b][k] (e.g. pic_compose's doc_offset)."""
    lib = load()
    g = geom._c()
    B, max_docs = req_doc_ids.shape
    if tuple(doc_target.shape) != (B, max_docs):
        raise ValueError("doc_target must be [batch][max_docs] like req_doc_ids")
    st = lib.pic_relocate(
        ctypes.byref(g), B, max_docs, doc_len.numel(), _ptr(k_pool, bf16, "k_pool"),
        _ptr(v_pool, bf16, "v_pool"), k_pool.shape[1],
        _ptr(doc_token_start, i64, "doc_token_start"), _ptr(doc_len, i32, "doc_len"),
        _ptr(doc_base_pos, i32, "doc_base_pos"), _ptr(req_doc_ids, i32, "req_doc_ids"),
        _ptr(req_num_docs, i32, "req_num_docs"), _ptr(doc_target, i32, "doc_target"),
        _ptr(block_table, i32, "block_table"), block_table.shape[1], num_pages,
        _ptr(k_cache, bf16, "k_cache"), _ptr(v_cache, bf16, "v_cache"), layer_begin, layer_end,
        _stream(stream))
    _check(st, "pic_relocate")


def pic_relocate_mapped(geom: Geometry, k_pool, v_pool, tok_map, doc_delta, slot_mapping,
                        num_pages: int, k_cache, v_cache, layer_begin: int, layer_end: int,
                        stream=None):
    """Relocation driven by pic_compose's token and slot maps."""
    lib = load()
    g = geom._c()
    B, max_docs = doc_delta.shape
    st = lib.pic_relocate_mapped(
        ctypes.byref(g), B, max_docs, _ptr(k_pool, bf16, "k_pool"), _ptr(v_pool, bf16, "v_pool"),
        k_pool.shape[1], _ptr(tok_map, i64, "tok_map"), _ptr(doc_delta, i32, "doc_delta"),
        _ptr(slot_mapping, i64, "slot_mapping"), slot_mapping.shape[1], num_pages,
        _ptr(k_cache, bf16, "k_cache"), _ptr(v_cache, bf16, "v_cache"), layer_begin, layer_end,
        _stream(stream))
    _check(st, "pic_relocate_mapped")


def pic_link(geom: Geometry, doc_len, doc_base_pos, doc_token_start, req_doc_ids, req_num_docs,
             prefix_len, query_len, block_table, num_pages: int, max_ctx: int, max_inline: int,
             k_pool, v_pool, layer_begin: int, layer_end: int, append_layer: int, q, k_new, v_new,
             inline_len, k_cache, v_cache, doc_offset, doc_delta, slot_mapping, tok_map, inline_pos,
             ctx_len, workspace, stream=None, span_len=None):
    """pic_compose + pic_relocate + pic_append_inline (append_layer, or none if < 0)
    in one launch; q/k_new/v_new are the append layer's inline projections;
    span_len as for pic_compose."""
    lib = load()
    g = geom._c()
    B, max_docs = req_doc_ids.shape
    app = append_layer >= 0
    st = lib.pic_link(
        ctypes.byref(g), B, max_docs, doc_len.numel(), _ptr(doc_len, i32, "doc_len"),
        _ptr(doc_base_pos, i32, "doc_base_pos"), _ptr(doc_token_start, i64, "doc_token_start"),
        _ptr(req_doc_ids, i32, "req_doc_ids"), _ptr(req_num_docs, i32, "req_num_docs"),
        _ptr(span_len, i32, "span_len", allow_none=True),
        _ptr(prefix_len, i32, "prefix_len"), _ptr(query_len, i32, "query_len"),
        _ptr(block_table, i32, "block_table"), block_table.shape[1], num_pages, max_ctx,
        max_inline, _ptr(k_pool, bf16, "k_pool"), _ptr(v_pool, bf16, "v_pool"), k_pool.shape[1],
        layer_begin, layer_end, append_layer, _ptr(q, bf16, "q", allow_none=not app),
        _ptr(k_new, bf16, "k_new", allow_none=not app), _ptr(v_new, bf16, "v_new", allow_none=not app),
        _ptr(inline_len, i32, "inline_len", allow_none=not app), _ptr(k_cache, bf16, "k_cache"),
        _ptr(v_cache, bf16, "v_cache"), _ptr(doc_offset, i32, "doc_offset"),
        _ptr(doc_delta, i32, "doc_delta"), _ptr(slot_mapping, i64, "slot_mapping"),
        _ptr(tok_map, i64, "tok_map"), _ptr(inline_pos, i32, "inline_pos"),
        _ptr(ctx_len, i32, "ctx_len"), _ptr(workspace, torch.uint8, "workspace", allow_none=not app),
        0 if workspace is None else workspace.numel(), _stream(stream))
    _check(st, "pic_link")


def pic_prefill_workspace_size(geom: Geometry, batch: int, max_inline: int, max_ctx: int,
                               num_splits: int = 0) -> int:
    g = geom._c()
    return load().pic_prefill_workspace_size(ctypes.byref(g), batch, max_inline, max_ctx,
                                             num_splits)


def pic_prefill_fused_workspace_size(geom: Geometry, batch: int, max_inline: int, max_ctx: int,
                                     max_docs: int, num_splits: int = 0) -> int:
    g = geom._c()
    return load().pic_prefill_fused_workspace_size(ctypes.byref(g), batch, max_inline, max_ctx,
                                                   max_docs, num_splits)


def pic_prefill_num_splits(geom: Geometry, batch: int, max_inline: int, max_ctx: int,
                           num_splits: int = 0) -> int:
    g = geom._c()
    return load().pic_prefill_num_splits(ctypes.byref(g), batch, max_inline, max_ctx, num_splits)


def pic_prefill_plan_splits(geom: Geometry, max_ctx: int, inline_len, inline_pos) -> int:
    """Key-split count planned from the requests' inline positions (host int32
    tensors [B] and [B][max_inline]); 0 on bad arguments."""
    import torch
    lens = inline_len.to(torch.int32).contiguous()
    pos = inline_pos.to(torch.int32).contiguous()
    if lens.is_cuda or pos.is_cuda or pos.dim() != 2 or lens.numel() != pos.shape[0]:
        raise ValueError("pic_prefill_plan_splits: host int32 inline_len [B] and inline_pos [B][T]")
    g = geom._c()
    return load().pic_prefill_plan_splits(ctypes.byref(g), pos.shape[0], pos.shape[1], max_ctx,
                                          ctypes.c_void_p(lens.data_ptr()),
                                          ctypes.c_void_p(pos.data_ptr()))


def pic_decode_num_splits(geom: Geometry, batch: int, max_ctx: int, num_splits: int = 0) -> int:
    g = geom._c()
    return load().pic_decode_num_splits(ctypes.byref(g), batch, max_ctx, num_splits)


def pic_append_inline(geom: Geometry, layer: int, q, k_new, v_new, inline_pos, inline_len,
                      slot_mapping, num_pages: int, k_cache, v_cache, workspace, stream=None):
    lib = load()
    g = geom._c()
    B, max_inline = inline_pos.shape
    st = lib.pic_append_inline(
        ctypes.byref(g), layer, B, max_inline, _ptr(q, bf16, "q"), _ptr(k_new, bf16, "k_new"),
        _ptr(v_new, bf16, "v_new"), _ptr(inline_pos, i32, "inline_pos"),
        _ptr(inline_len, i32, "inline_len"), _ptr(slot_mapping, i64, "slot_mapping"),
        slot_mapping.shape[1], num_pages, _ptr(k_cache, bf16, "k_cache"),
        _ptr(v_cache, bf16, "v_cache"), _ptr(workspace, torch.uint8, "workspace"),
        workspace.numel(), _stream(stream))
    _check(st, "pic_append_inline")


def _projections(q, k_new, v_new):
    given = [t is not None for t in (q, k_new, v_new)]
    if any(given) and not all(given):
        raise ValueError("give q, k_new and v_new together, or none")
    return (_ptr(q, bf16, "q", allow_none=True), _ptr(k_new, bf16, "k_new", allow_none=True),
            _ptr(v_new, bf16, "v_new", allow_none=True))


def pic_attend_prefill(geom: Geometry, layer: int, inline_pos, inline_len, max_ctx: int,
                       block_table, num_pages: int, k_cache, v_cache, out, lse=None,
                       num_splits: int = 0, workspace=None, stream=None, q=None, k_new=None,
                       v_new=None):
    """Prefill attention of one layer.  With q, k_new and v_new (the layer's
    un-rotated inline projections) the call appends them itself first;
    without, the workspace must hold this layer's append (pic_append_inline
    or pic_link)."""
    lib = load()
    g = geom._c()
    B, max_inline = inline_pos.shape
    st = lib.pic_attend_prefill(
        ctypes.byref(g), layer, B, max_inline, *_projections(q, k_new, v_new),
        _ptr(inline_pos, i32, "inline_pos"),
        _ptr(inline_len, i32, "inline_len"), max_ctx, _ptr(block_table, i32, "block_table"),
        block_table.shape[1], num_pages, _ptr(k_cache, bf16, "k_cache"),
        _ptr(v_cache, bf16, "v_cache"), _ptr_or_pinned(out, bf16, "out"),
        _ptr(lse, f32, "lse", allow_none=True), num_splits,
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream))
    _check(st, "pic_attend_prefill")


def pic_attend_prefill_fused(geom: Geometry, layer: int, inline_pos, inline_len, max_ctx: int,
                             block_table, num_pages: int, k_cache, v_cache, k_pool, v_pool,
                             tok_map, doc_delta, out, lse=None, num_splits: int = 0,
                             workspace=None, stream=None, q=None, k_new=None, v_new=None):
    """Rotate-on-load prefill attention: documents read from the pool and
    rotated as they are loaded (tok_map / doc_delta from pic_compose); q,
    k_new, v_new as for pic_attend_prefill."""
    lib = load()
    g = geom._c()
    B, max_inline = inline_pos.shape
    max_docs = doc_delta.shape[1]
    if tuple(tok_map.shape) != (B, max_ctx):
        raise ValueError("tok_map must be [batch][max_ctx]")
    st = lib.pic_attend_prefill_fused(
        ctypes.byref(g), layer, B, max_inline, *_projections(q, k_new, v_new),
        _ptr(inline_pos, i32, "inline_pos"), _ptr(inline_len, i32, "inline_len"), max_ctx,
        _ptr(block_table, i32, "block_table"), block_table.shape[1], num_pages,
        _ptr(k_cache, bf16, "k_cache"), _ptr(v_cache, bf16, "v_cache"),
        _ptr(k_pool, bf16, "k_pool"), _ptr(v_pool, bf16, "v_pool"), k_pool.shape[1], max_docs,
        _ptr(tok_map, i64, "tok_map"), _ptr(doc_delta, i32, "doc_delta"),
        _ptr_or_pinned(out, bf16, "out"), _ptr(lse, f32, "lse", allow_none=True), num_splits,
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream))
    _check(st, "pic_attend_prefill_fused")


def pic_decode_workspace_size(geom: Geometry, batch: int, max_ctx: int, num_splits: int = 0) -> int:
    g = geom._c()
    return load().pic_decode_workspace_size(ctypes.byref(g), batch, max_ctx, num_splits)


def pic_attend_decode(geom: Geometry, layer: int, q, k_new, v_new, pos, block_table,
                      num_pages: int, k_cache, v_cache, out, max_ctx: int, lse=None,
                      num_splits: int = 0, workspace=None, pos_offset: int = 0, stream=None):
    lib = load()
    g = geom._c()
    B = pos.numel()
    st = lib.pic_attend_decode(
        ctypes.byref(g), layer, B, _ptr(q, bf16, "q"), _ptr(k_new, bf16, "k_new"),
        _ptr(v_new, bf16, "v_new"), _ptr(pos, i32, "pos"), pos_offset,
        _ptr(block_table, i32, "block_table"),
        block_table.shape[1], num_pages, _ptr(k_cache, bf16, "k_cache"),
        _ptr(v_cache, bf16, "v_cache"), _ptr(out, bf16, "out"),
        _ptr(lse, f32, "lse", allow_none=True), max_ctx, num_splits,
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream))
    _check(st, "pic_attend_decode")


def pic_attend_decode_noalloc(geom: Geometry, layer: int, q, k_new, v_new, pos, block_table,
                              num_pages: int, k_cache, v_cache, out, max_ctx: int, lse=None,
                              num_splits: int = 0, pos_offset: int = 0, stream=None):
    """pic_attend_decode without a workspace, for callers that cannot allocate
    while decoding; the scratch is an array inside the library (see pic.h)."""
    lib = load()
    g = geom._c()
    B = pos.numel()
    st = lib.pic_attend_decode_noalloc(
        ctypes.byref(g), layer, B, _ptr(q, bf16, "q"), _ptr(k_new, bf16, "k_new"),
        _ptr(v_new, bf16, "v_new"), _ptr(pos, i32, "pos"), pos_offset,
        _ptr(block_table, i32, "block_table"), block_table.shape[1], num_pages,
        _ptr(k_cache, bf16, "k_cache"), _ptr(v_cache, bf16, "v_cache"), _ptr(out, bf16, "out"),
        _ptr(lse, f32, "lse", allow_none=True), max_ctx, num_splits, _stream(stream))
    _check(st, "pic_attend_decode_noalloc")


def pic_attention_deviation(geom: Geometry, layer: int, inline_pos, inline_len, query_len,
                            req_doc_ids, doc_len, doc_offset, slot_mapping,
                            num_pages: int, k_cache_a, k_cache_b, lse_a, lse_b, workspace,
                            sums, counts, edges=(0.0, 0.1, 0.9), max_query_len=None,
                            stream=None):
    """D_r(A, B) of two stitched key caches (see include/pic.h): fills
    sums [B][R] (float64) and counts [B][R] (int64) for the regions between
    consecutive ``edges``."""
    lib = load()
    g = geom._c()
    B, max_inline = inline_pos.shape
    if max_query_len is None:
        max_query_len = int(query_len.max().item())
    arr = (ctypes.c_double * len(edges))(*[float(e) for e in edges])
    st = lib.pic_attention_deviation(
        ctypes.byref(g), layer, B, max_inline, req_doc_ids.shape[1], slot_mapping.shape[1],
        num_pages, _ptr(inline_pos, i32, "inline_pos"), _ptr(inline_len, i32, "inline_len"),
        _ptr(query_len, i32, "query_len"), int(max_query_len), _ptr(req_doc_ids, i32, "req_doc_ids"),
        _ptr(doc_len, i32, "doc_len"), _ptr(doc_offset, i32, "doc_offset"),
        _ptr(slot_mapping, i64, "slot_mapping"),
        _ptr(k_cache_a, bf16, "k_cache_a"), _ptr(k_cache_b, bf16, "k_cache_b"),
        _ptr(lse_a, f32, "lse_a"), _ptr(lse_b, f32, "lse_b"), ctypes.cast(arr, ctypes.c_void_p),
        len(edges) - 1,
        _ptr(workspace, torch.uint8, "workspace"), workspace.numel(),
        _ptr(sums, torch.float64, "sums"), _ptr(counts, i64, "counts"), _stream(stream))
    _check(st, "pic_attention_deviation")
