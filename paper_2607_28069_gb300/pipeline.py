"""The cache-hit path over one workload: device buffers plus the call sequence.

compose -> relocate (all layers) -> per layer: prefill (inline append +
attention) -> decode steps.  PyTorch only allocates device memory and
supplies the stream; every step is a libpic call.
"""
from __future__ import annotations

import torch

from . import (Geometry, pic_append_inline, pic_attend_decode, pic_attend_prefill,
               pic_attend_prefill_fused, pic_compose, pic_copy_async, pic_decode_workspace_size,
               pic_link, pic_prefill_fused_workspace_size, pic_prefill_plan_splits, pic_relocate,
               pic_relocate_mapped)
from .workloads import Workload


def host_inline_positions(wl: Workload):
    """The inline tokens' logical positions of every request, on the host:
    the prefix from 0, each document's span right after the document, the
    query after the last one (the canonical order P, D_1, S_1, ..., D_m, S_m,
    Q that compose lays out).  For planning only; compose computes the
    positions the kernels use, and reports malformed requests, for which
    this returns None."""
    B = wl.req_doc_ids.shape[0]
    prefix, query = wl.prefix_len.cpu().tolist(), wl.query_len.cpu().tolist()
    ndocs, ids = wl.req_num_docs.cpu().tolist(), wl.req_doc_ids.cpu().tolist()
    dlen = wl.doc_len.cpu().tolist()
    spans = wl.span_len.cpu().tolist() if wl.span_len is not None else None
    pos = torch.zeros((B, wl.tin_max), dtype=torch.int32)
    lens = torch.zeros((B,), dtype=torch.int32)
    for b in range(B):
        if not 0 <= ndocs[b] <= len(ids[b]) or prefix[b] < 0 or query[b] < 0:
            return None
        row = list(range(prefix[b]))
        off = prefix[b]
        for k in range(ndocs[b]):
            if not 0 <= ids[b][k] < len(dlen):
                return None
            off += dlen[ids[b][k]]
            s_k = spans[b][k] if spans is not None else 0
            row += range(off, off + s_k)
            off += s_k
        row += range(off, off + query[b])
        row = row[:wl.tin_max]
        pos[b, :len(row)] = torch.tensor(row, dtype=torch.int32)
        lens[b] = len(row)
    return lens, pos


class CacheHitPath:
    def __init__(self, wl: Workload, prefill_splits: int = 0, decode_splits: int = 0,
                 with_lse: bool = False, rope_style: int = 0, inv_freq=None,
                 layer_inv_freq=None):
        spec = wl.spec
        dev = wl.k_pool.device
        self.wl = wl
        self.geom = Geometry(spec.layers, spec.q_heads, spec.kv_heads, spec.head_dim,
                             spec.rope_base, page_size=spec.page_size, rope_style=rope_style,
                             inv_freq=inv_freq, layer_inv_freq=layer_inv_freq)
        B, md = wl.req_doc_ids.shape
        L, Hq, Hkv, d = spec.layers, spec.q_heads, spec.kv_heads, spec.head_dim
        self.B, self.max_docs = B, md
        self.max_ctx = wl.max_ctx
        self.max_inline = wl.tin_max
        if prefill_splits == 0:  # planned from the requests' layout (else the library's choice)
            hp = host_inline_positions(wl)
            if hp is not None:
                prefill_splits = pic_prefill_plan_splits(self.geom, self.max_ctx, *hp)
        self.prefill_splits = prefill_splits
        self.decode_splits = decode_splits
        i32, i64, bf16 = torch.int32, torch.int64, torch.bfloat16
        self.doc_offset = torch.empty((B, md), dtype=i32, device=dev)
        self.doc_delta = torch.empty((B, md), dtype=i32, device=dev)
        self.slot_mapping = torch.empty((B, self.max_ctx), dtype=i64, device=dev)
        self.tok_map = torch.empty((B, self.max_ctx), dtype=i64, device=dev)
        self.inline_pos = torch.empty((B, self.max_inline), dtype=i32, device=dev)
        self.ctx_len = torch.empty((B,), dtype=i32, device=dev)
        shape = (L, wl.num_pages, Hkv, spec.page_size, d)
        self.k_cache = torch.zeros(shape, dtype=bf16, device=dev)
        self.v_cache = torch.zeros(shape, dtype=bf16, device=dev)
        u8 = torch.uint8
        # one prefill workspace for the materialised and the rotate-on-load
        # calls (the latter's is the larger)
        self.ws_prefill = torch.empty(
            pic_prefill_fused_workspace_size(self.geom, B, self.max_inline, self.max_ctx, md,
                                             prefill_splits),
            dtype=u8, device=dev)
        self.out = torch.empty((L, B, self.max_inline, Hq, d), dtype=bf16, device=dev)
        self.lse = torch.empty((L, B, self.max_inline, Hq), dtype=torch.float32,
                               device=dev) if with_lse else None
        self.dec_out = self.dec_lse = self.ws_decode = None
        self._request_dev = None
        if wl.q_dec is not None:
            self.ws_decode = torch.empty(
                pic_decode_workspace_size(self.geom, B, self.max_ctx, decode_splits),
                dtype=u8, device=dev)
            self.dec_out = torch.empty((L, B, Hq, d), dtype=bf16, device=dev)
            self.dec_lse = torch.empty((L, B, Hq), dtype=torch.float32,
                                       device=dev) if with_lse else None

    # -- per-request inputs as one upload
    REQUEST_FIELDS = ("req_doc_ids", "req_num_docs", "prefix_len", "query_len", "block_table",
                      "inline_len")
    LAYER_FIELDS = ("q_inline", "k_inline", "v_inline")

    def pack_request_inputs(self) -> torch.Tensor:
        """Move the per-request inputs (document choice, lengths, block table,
        inline projections) into one contiguous device buffer, rebinding the
        workload's tensors to views of it, and return a pinned host mirror
        holding the same bytes.  A serving loop then writes a request into
        the mirror and calls ``upload`` once: one host-to-device copy per
        step instead of one per tensor.  The document pool stays resident.

        Layout: the per-request fields first, then layer by layer that
        layer's q, k and v, so that the bytes layer 0 needs are one prefix
        and each later layer one contiguous range (``served_pass`` streams
        them)."""
        wl = self.wl
        L = wl.spec.layers
        align = lambda n: (n + 255) // 256 * 256  # noqa: E731
        fields = self.REQUEST_FIELDS + (("span_len",) if wl.span_len is not None else ())
        offs, total = [], 0
        for name in fields:
            t = getattr(wl, name)
            offs.append(total)
            total += align(t.numel() * t.element_size())
        per_layer = [align(getattr(wl, f)[0].numel() * 2) for f in self.LAYER_FIELDS]
        layer0 = total
        layer_bytes = sum(per_layer)
        total += L * layer_bytes
        dev = torch.empty(total, dtype=torch.uint8, device=wl.k_pool.device)
        host = torch.empty(total, dtype=torch.uint8, pin_memory=True)
        for name, off in zip(fields, offs):
            t = getattr(wl, name)
            n = t.numel() * t.element_size()
            view = dev[off:off + n].view(t.dtype).view(t.shape)
            view.copy_(t)
            setattr(wl, name, view)
        buf16 = dev.view(torch.bfloat16)
        off = layer0
        for f, nb in zip(self.LAYER_FIELDS, per_layer):
            t = getattr(wl, f)
            assert t.dtype == torch.bfloat16 and t.is_contiguous()
            view = torch.as_strided(buf16, t.shape, (layer_bytes // 2,) + t.stride()[1:], off // 2)
            view.copy_(t)
            setattr(wl, f, view)
            off += nb
        host.copy_(dev.cpu())
        self._request_dev = dev
        self._layer_ranges = [(layer0 + l * layer_bytes, layer0 + (l + 1) * layer_bytes)
                              for l in range(L)]
        return host

    def upload(self, host: torch.Tensor):
        """One asynchronous copy of a packed request (see pack_request_inputs),
        moved by the library's copy kernel (pic_copy_async)."""
        pic_copy_async(self._request_dev, host)

    def download(self, host_out: torch.Tensor, dev: torch.Tensor | None = None):
        """Asynchronous copy of the attention outputs (or `dev`) into the pinned
        host tensor host_out, by the library's copy kernel."""
        pic_copy_async(host_out, self.out if dev is None else dev)

    def served_pass(self, host: torch.Tensor, host_out: torch.Tensor,
                    up_stream: torch.cuda.Stream, down_stream: torch.cuda.Stream):
        """One TTFT pass (as ``ttft_pass``) with the request's inputs taken
        from the pinned host mirror ``host`` and every layer's attention
        output written to the pinned ``host_out`` [L][B][T][Hq][d], the
        copies overlapping the compute: the per-request fields go first (copy
        kernel), then the link runs without its append (layout and every
        layer's relocation need no projections) while layer 0's projections
        arrive on ``up_stream`` by the copy kernel and those of layers 1..
        follow by the copy engine; layer l's append waits for its range.
        The output of each layer but the last streams out on
        ``down_stream`` once its attention is done; the last layer's
        attention writes its rows into ``host_out`` itself (pinned host
        memory, reached over the chip-to-chip link).  Returns with the current stream
        ordered after every copy.  Capturable in a CUDA graph."""
        L = self.wl.spec.layers
        main = torch.cuda.current_stream()
        dev = self._request_dev
        fields_end = self._layer_ranges[0][0]
        pic_copy_async(dev[:fields_end], host[:fields_end])
        up_stream.wait_stream(main)
        down_stream.wait_stream(main)
        up_done = []
        with torch.cuda.stream(up_stream):
            for l in range(L):
                lo, hi = self._layer_ranges[l]
                if l == 0:
                    pic_copy_async(dev[lo:hi], host[lo:hi])
                else:
                    dev[lo:hi].copy_(host[lo:hi], non_blocking=True)
                up_done.append(torch.cuda.Event())
                up_done[l].record(up_stream)
        for l in range(L):
            if l == 0:
                self.link(-1)
            main.wait_event(up_done[l])
            self.append(l)
            if l < L - 1:
                self.attend(l)
                down_stream.wait_stream(main)
                with torch.cuda.stream(down_stream):
                    host_out[l].copy_(self.out[l], non_blocking=True)
            else:
                self.attend(l, out=host_out[l])  # the last layer's rows go straight to the host
        main.wait_stream(up_stream)
        main.wait_stream(down_stream)

    # -- a1: layout and slot map
    def compose(self):
        wl = self.wl
        pic_compose(self.geom, wl.doc_len, wl.doc_base_pos, wl.doc_token_start, wl.req_doc_ids,
                    wl.req_num_docs, wl.prefix_len, wl.query_len, wl.block_table, wl.num_pages,
                    self.max_ctx, self.max_inline, self.doc_offset, self.doc_delta,
                    self.slot_mapping, self.tok_map, self.inline_pos, self.ctx_len,
                    span_len=wl.span_len)

    # -- a2 + a3: per-document rotation and stitching, all layers, one launch:
    # every document from its base position to the target compose assigned
    def relocate(self, layer_begin: int = 0, layer_end: int | None = None):
        wl = self.wl
        if layer_end is None:
            layer_end = wl.spec.layers
        pic_relocate(self.geom, wl.k_pool, wl.v_pool, wl.doc_token_start, wl.doc_len,
                     wl.doc_base_pos, wl.req_doc_ids, wl.req_num_docs, self.doc_offset,
                     wl.block_table, wl.num_pages, self.k_cache, self.v_cache, layer_begin,
                     layer_end)

    # -- the same through compose's token and slot maps
    def relocate_mapped(self, layer_begin: int = 0, layer_end: int | None = None):
        wl = self.wl
        if layer_end is None:
            layer_end = wl.spec.layers
        pic_relocate_mapped(self.geom, wl.k_pool, wl.v_pool, self.tok_map, self.doc_delta,
                            self.slot_mapping, wl.num_pages, self.k_cache, self.v_cache,
                            layer_begin, layer_end)

    # -- a1 + a2 + a3 + a4 (first layer) in one launch
    def link(self, append_layer: int = 0):
        wl = self.wl
        L = wl.spec.layers
        app = append_layer >= 0
        pic_link(self.geom, wl.doc_len, wl.doc_base_pos, wl.doc_token_start, wl.req_doc_ids,
                 wl.req_num_docs, wl.prefix_len, wl.query_len, wl.block_table, wl.num_pages,
                 self.max_ctx, self.max_inline, wl.k_pool, wl.v_pool, 0, L, append_layer,
                 wl.q_inline[append_layer] if app else None,
                 wl.k_inline[append_layer] if app else None,
                 wl.v_inline[append_layer] if app else None, wl.inline_len if app else None,
                 self.k_cache, self.v_cache, self.doc_offset, self.doc_delta, self.slot_mapping,
                 self.tok_map, self.inline_pos, self.ctx_len, self.ws_prefill if app else None,
                 span_len=wl.span_len)

    # -- a4: RoPE + append of the inline tokens of one layer
    def append(self, layer: int):
        wl = self.wl
        pic_append_inline(self.geom, layer, wl.q_inline[layer], wl.k_inline[layer],
                          wl.v_inline[layer], self.inline_pos, wl.inline_len, self.slot_mapping,
                          wl.num_pages, self.k_cache, self.v_cache, self.ws_prefill)

    # -- a5: prefill attention of one layer
    def attend(self, layer: int, out: torch.Tensor | None = None):
        """Prefill attention of one layer into self.out[layer], or into `out`
        (for instance a pinned host tensor, written by the kernels directly)."""
        wl = self.wl
        pic_attend_prefill(self.geom, layer, self.inline_pos, wl.inline_len, self.max_ctx,
                           wl.block_table, wl.num_pages, self.k_cache, self.v_cache,
                           self.out[layer] if out is None else out,
                           None if self.lse is None else self.lse[layer],
                           self.prefill_splits, self.ws_prefill)

    # -- a7: prefill attention reading the documents from the pool (no relocate)
    def attend_fused(self, layer: int, out: torch.Tensor | None = None):
        """Rotate-on-load attention of one layer (the workspace holds the
        layer's append); `out` as for attend."""
        wl = self.wl
        pic_attend_prefill_fused(self.geom, layer, self.inline_pos, wl.inline_len, self.max_ctx,
                                 wl.block_table, wl.num_pages, self.k_cache, self.v_cache,
                                 wl.k_pool, wl.v_pool, self.tok_map, self.doc_delta,
                                 self.out[layer] if out is None else out,
                                 None if self.lse is None else self.lse[layer],
                                 self.prefill_splits, self.ws_prefill)

    def prefill(self, layer: int):
        """Append and attention of one layer: one pic_attend_prefill call
        given the layer's projections (the same launches as append then
        attend)."""
        wl = self.wl
        pic_attend_prefill(self.geom, layer, self.inline_pos, wl.inline_len, self.max_ctx,
                           wl.block_table, wl.num_pages, self.k_cache, self.v_cache,
                           self.out[layer], None if self.lse is None else self.lse[layer],
                           self.prefill_splits, self.ws_prefill, q=wl.q_inline[layer],
                           k_new=wl.k_inline[layer], v_new=wl.v_inline[layer])

    def fused_pass(self):
        """The cache-hit path with rotate-on-load attention: layout, then per
        layer the inline append and the fused attention; no relocation."""
        self.compose()
        for layer in range(self.wl.spec.layers):
            self.append(layer)
            self.attend_fused(layer)

    # -- a6: one decode step of one layer (token position ctx_len + step)
    def decode(self, step: int, layer: int):
        wl = self.wl
        pic_attend_decode(self.geom, layer, wl.q_dec[step, layer], wl.k_dec[step, layer],
                          wl.v_dec[step, layer], self.ctx_len, wl.block_table, wl.num_pages,
                          self.k_cache, self.v_cache, self.dec_out[layer], self.max_ctx,
                          None if self.dec_lse is None else self.dec_lse[layer],
                          self.decode_splits, self.ws_decode, pos_offset=step)

    def ttft_pass(self, linked: bool = True):
        """The cache-hit path up to the first token: layout, re-rotation and
        stitching of every layer, then every layer's inline prefill.  With
        ``linked`` the layout, the relocation and the first layer's inline
        append are one pic_link launch; otherwise the separate calls."""
        if linked:
            self.link(0)
            self.attend(0)
            first = 1
        else:
            self.compose()
            self.relocate()
            first = 0
        for layer in range(first, self.wl.spec.layers):
            self.prefill(layer)

    def decode_pass(self, step: int):
        for layer in range(self.wl.spec.layers):
            self.decode(step, layer)
