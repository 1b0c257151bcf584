/*
 * pic.h -- C ABI of the GB300 (sm_103a) cache-hit path of SemPIC-style
 * position-independent KV caching.
 *
 * The path (SemPIC, "Cache-hit serving"; appendix "Position-Independent
 * Linking"): cached document keys, compiled in isolation at a base position,
 * are moved to their request-time logical positions with the key re-rotation
 * of Eq. 3, stitched with the request's inline tokens into a paged KV cache in
 * the canonical order P, D_1..D_m, Q (Eqs. 1-2), and read by the unchanged
 * decoder's GQA softmax attention under the frontier causal mask, first for
 * the inline tokens (prefill) and then for ordinary decoding.
 *
 * Conventions shared by every call
 * --------------------------------
 * - Every tensor pointer is DEVICE memory owned by the caller, except where a
 *   call says it may also be page-locked host memory (pic_copy_async, the
 *   output of pic_attend_prefill); the library allocates nothing and keeps no
 *   pointer after a call returns.
 * - Every call is asynchronous on `stream` (NULL = legacy default stream).
 *   Outputs are valid once the stream has reached the call.
 * - bf16 tensors are IEEE bfloat16, row-major, densely packed, in the layouts
 *   given per argument.  Integer tensors are int32 unless noted.
 * - Host-side argument checks return PIC_ERR_INVALID_ARG / PIC_ERR_UNSUPPORTED
 *   before anything is launched.  Checks that need device data (document ids,
 *   page ids, positions, lengths) run inside the kernels: a failing element is
 *   skipped (never dereferenced) and the first failure is recorded in a
 *   per-device status word read by pic_device_status().  Every wait inside a
 *   kernel is bounded; expiry is recorded as PIC_DEV_TIMEOUT.
 * - On a non-OK return, pic_last_error() gives a one-line reason (per thread).
 * - No call throws; no call synchronises the stream except pic_device_status.
 *
 * Cache layout (all calls): k_cache / v_cache are
 *     bf16 [num_layers][num_pages][num_kv_heads][page_size][head_dim]
 * Logical position t of request b lives in page block_table[b][t / page_size]
 * at row t % page_size ("slot" = page * page_size + row).
 * Document pool layout: k_pool / v_pool are
 *     bf16 [num_layers][pool_tokens][num_kv_heads][head_dim]
 * document i occupying rows doc_token_start[i] .. + doc_len[i] - 1, its key
 * at row j compiled at logical position doc_base_pos[i] + j.
 */
#ifndef PIC_H_
#define PIC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define PIC_ABI_VERSION 4

typedef struct CUstream_st *pic_stream_t; /* identical to cudaStream_t */

typedef enum {
  PIC_OK = 0,
  PIC_ERR_INVALID_ARG = 1, /* a host-visible argument is out of range       */
  PIC_ERR_UNSUPPORTED = 2, /* valid but not implemented (head_dim, page)    */
  PIC_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed             */
  PIC_ERR_WORKSPACE = 4,   /* workspace missing, too small or misaligned    */
  PIC_ERR_DEVICE = 5       /* pic_device_status found a device-side failure */
} pic_status_t;

/* Device-side failure codes reported by pic_device_status(). */
#define PIC_DEV_OK 0
#define PIC_DEV_BAD_DOC_ID 1        /* request names a doc outside the pool  */
#define PIC_DEV_BAD_DOC_LEN 2       /* document length <= 0                  */
#define PIC_DEV_BAD_REQUEST 3       /* negative prefix/query/doc count       */
#define PIC_DEV_CTX_OVERFLOW 4      /* context exceeds max_ctx / max_inline  */
#define PIC_DEV_BLOCK_TABLE_SHORT 5 /* block table has too few pages         */
#define PIC_DEV_BAD_PAGE 6          /* page id outside [0, num_pages)        */
#define PIC_DEV_BAD_POSITION 7      /* logical position out of range         */
#define PIC_DEV_TIMEOUT 8           /* a bounded wait inside a kernel expired */

/* RoPE pairing: element i with i + d/2 (half-split), or 2i with 2i+1. */
#define PIC_ROPE_HALF 0
#define PIC_ROPE_INTERLEAVED 1

/* Model geometry shared by all calls. */
typedef struct {
  int32_t num_layers;
  int32_t num_q_heads;   /* Hq; query head h reads kv head h / (Hq / Hkv)  */
  int32_t num_kv_heads;  /* Hkv; must divide Hq                            */
  int32_t head_dim;      /* d: 64 or 128                                   */
  int32_t page_size;     /* tokens per page: 16                            */
  int32_t rope_style;    /* PIC_ROPE_HALF or PIC_ROPE_INTERLEAVED          */
  double rope_base;      /* theta_i = rope_base^(-2i/d)                    */
  const double *inv_freq;/* nullable HOST pointer to d/2 frequencies that
                            replace rope_base^(-2i/d) (scaled RoPE)        */
  const double *layer_inv_freq; /* nullable DEVICE pointer to [num_layers][d/2]
                            frequencies, row l for layer l (a layer-specific
                            rotary transform R_l, Eq. 3); overrides rope_base
                            and inv_freq.  Values must be positive and finite
                            (not checked); the caller keeps it alive while
                            calls that use the geometry run.             */
} pic_geom_t;

/* Library version (PIC_ABI_VERSION of the build). */
int32_t pic_abi_version(void);

/* One-line reason for the last non-OK status returned on this thread. */
const char *pic_last_error(void);

/*
 * pic_device_status -- synchronise `stream`, then read and clear the status
 * word of the current device.  *code receives a PIC_DEV_* value, *detail the
 * request (or split) index of the first failure.  Returns PIC_ERR_DEVICE when
 * *code != PIC_DEV_OK, PIC_ERR_CUDA when the synchronisation failed.
 */
pic_status_t pic_device_status(pic_stream_t stream, int32_t *code, int32_t *detail);

/*
 * pic_copy_async -- copy `bytes` from src to dst on `stream`, where each of
 * src and dst is memory of the current device or page-locked host memory
 * (cudaHostAlloc, cudaHostRegister, a pinned torch tensor).  Not an
 * operation of the paper: the transfer of a request's inputs and outputs
 * that a serving loop performs around the cache-hit path.  The bytes are
 * moved by a kernel (16-byte loads and stores; host memory is reached over
 * the chip-to-chip link of a Grace-Blackwell node), which for transfers of a
 * few megabytes is faster than the copy engines; when either address is not
 * 16-byte aligned the copy engine moves them instead.  Asynchronous: the
 * caller keeps both buffers alive and unmodified until the stream reaches
 * the copy.  Errors: PIC_ERR_INVALID_ARG for NULL, pageable host memory,
 * another device's memory or overlapping ranges; bytes = 0 does nothing.
 */
pic_status_t pic_copy_async(void *dst, const void *src, size_t bytes, pic_stream_t stream);

/*
 * pic_launch_probe -- a measurement aid, not an operation of the paper: n
 * empty kernels launched in order on `stream`, each a programmatic dependent
 * of the one before (as every kernel of the path is), with grid
 * grid[3i .. 3i+2], block[i] threads and smem[i] bytes of dynamic shared
 * memory.  Timing a chain with the launch shapes of a pass gives the part of
 * that pass no kernel work can remove: launch, dependency and CTA
 * scheduling.  PIC_ERR_INVALID_ARG for sizes out of range (block > 1024,
 * shared memory above the device's opt-in limit).
 */
pic_status_t pic_launch_probe(int32_t n, const int32_t *grid, const int32_t *block,
                              const int32_t *smem, pic_stream_t stream);

/*
 * pic_wait_probe -- a check of the failure detection, not an operation of the
 * paper: one CTA of one warp waits on the first phase of an mbarrier of one
 * arrival with the bounded wait every kernel of the path uses, limited to
 * limit_ns.  arrive != 0: the CTA arrives first and the wait completes at
 * once.  arrive == 0: nothing arrives; after limit_ns the wait records
 * PIC_DEV_TIMEOUT (detail -1) in the status word read by pic_device_status
 * and the kernel returns, so the context stays usable.  Asynchronous on
 * `stream`.  PIC_ERR_INVALID_ARG for limit_ns outside [1000, 10^10].
 */
pic_status_t pic_wait_probe(int32_t arrive, int64_t limit_ns, pic_stream_t stream);

/*
 * pic_compose -- link operator R: logical layout of each request and its
 * token-level maps (Eqs. 1-2, "Background: Position-Independent Caching";
 * appendix "Logical Layout and Re-Rotation").
 *
 * Request b is laid out in the canonical order P, D_1, S_1, ..., D_m, S_m, Q
 * (Eq. 1): the prefix (positions 0..P_b-1), then for k = 0..m_b-1 its k-th
 * document (order req_doc_ids[b][..]) followed by that document's inline
 * span of s_bk = span_len[b][k] tokens (a request-time span computed online,
 * not a cached block; span_len NULL: every s_bk = 0), then Tq_b query
 * tokens.  For its k-th document (pool id i, length n_i):
 *     doc_offset[b][k] = P_b + sum_{k'<k} (n_{ids[b][k']} + s_bk')
 *     doc_delta[b][k]  = doc_offset[b][k] - doc_base_pos[i]
 * ctx_len[b] = P_b + sum_k (n + s_bk) + Tq_b, and for 0 <= t < ctx_len[b]
 *     slot_mapping[b][t] = block_table[b][t / page] * page + t % page
 *     tok_map[b][t] = (k << 40) | (doc_token_start[i] + t - doc_offset[b][k])
 *                     for a position t of the k-th document, -1 otherwise
 * (the source row in the pool and the document index of every position).
 * inline_pos[b][0..T_b-1], T_b = P_b + sum_k s_bk + Tq_b, lists the inline
 * tokens' logical positions in this order: 0..P_b-1, then the positions of
 * each span (doc_offset[b][k] + n .. + s_bk - 1, k ascending), then
 * ctx_len[b]-Tq_b .. ctx_len[b]-1.  The inline projections that
 * pic_append_inline and pic_link take are in the same order.
 *
 * Inputs (device): doc_len, doc_base_pos int32 [n_pool_docs]; doc_token_start
 *   int64 [n_pool_docs]; req_doc_ids int32 [batch][max_docs]; span_len int32
 *   [batch][max_docs] or NULL; req_num_docs, prefix_len, query_len int32
 *   [batch]; block_table int32 [batch][max_pages] (entries used must be in
 *   [0, num_pages)).  max_docs <= 8192.
 * Outputs (device): doc_offset, doc_delta int32 [batch][max_docs] (entries
 *   k >= m_b are set to -1 / 0); slot_mapping, tok_map int64 [batch][max_ctx]
 *   (-1 beyond ctx_len); inline_pos int32 [batch][max_inline] (unused tail -1);
 *   ctx_len int32 [batch] (-1 for a request that failed a device check).
 * Device checks: doc id range, doc length > 0, span length >= 0,
 *   ctx <= max_ctx, T_b <= max_inline, ceil(ctx / page) <= max_pages, page ids
 *   in range.
 */
pic_status_t pic_compose(const pic_geom_t *geom, int32_t batch, int32_t max_docs,
                         int32_t n_pool_docs, const int32_t *doc_len,
                         const int32_t *doc_base_pos, const int64_t *doc_token_start,
                         const int32_t *req_doc_ids, const int32_t *req_num_docs,
                         const int32_t *span_len, const int32_t *prefix_len,
                         const int32_t *query_len,
                         const int32_t *block_table, int32_t max_pages, int64_t num_pages,
                         int32_t max_ctx, int32_t max_inline, int32_t *doc_offset,
                         int32_t *doc_delta, int64_t *slot_mapping, int64_t *tok_map,
                         int32_t *inline_pos, int32_t *ctx_len, pic_stream_t stream);

/*
 * pic_relocate -- key re-rotation and stitching of the cached documents
 * (Eq. 3, "Background: Position-Independent Caching"; appendix "Logical
 * Layout and Re-Rotation": only keys are rotated, values are reused as they
 * are).  The arguments are the problem as the paper states it: per document
 * its prepared KV block (pool rows), base position and target position.
 *
 * For every layer l in [layer_begin, layer_end), request b and its k-th
 * listed document (k < req_num_docs[b], pool id i = req_doc_ids[b][k],
 * n_i = doc_len[i] tokens, compiled at base position a_i = doc_base_pos[i])
 * placed at target position t_bk = doc_target[b][k], each token j < n_i:
 *     k_cache[l][slot(t_bk + j)] = R(t_bk - a_i) * k_pool[l][doc_token_start[i] + j]
 *     v_cache[l][slot(t_bk + j)] = v_pool[l][doc_token_start[i] + j]   (bit copy)
 * with slot(t) = block_table[b][t / page] * page + t % page.  R(delta)
 * rotates each RoPE pair by delta * theta_i: moving a key from a + j to
 * t + j is R(t + j) R(a + j)^-1 = R(t - a), one rotation per document.
 * cos/sin come from the angle formed and reduced in fp64; the rotation is
 * fp32; K' is rounded to bf16 (round to nearest even).  delta == 0
 * reproduces k bit-exactly.  The canonical placement of pic_compose is
 * doc_target = its doc_offset output, but any placement is accepted.
 *
 * Inputs (device): k_pool, v_pool (pool layout above) with pool_tokens rows
 *   per layer; doc_token_start int64, doc_len, doc_base_pos int32
 *   [n_pool_docs]; req_doc_ids, doc_target int32 [batch][max_docs];
 *   req_num_docs int32 [batch]; block_table int32 [batch][max_pages].
 * Device checks (pic_device_status; the failing document is skipped):
 *   document id outside the pool, length <= 0 or rows past the pool,
 *   negative target, target + n beyond max_pages pages, a page id outside
 *   [0, num_pages); two documents of a request whose target ranges overlap
 *   are reported as PIC_DEV_BAD_POSITION (both are still written, so the
 *   overlap holds one of them).
 * One launch, no workspace.  max_docs == 0 returns PIC_OK without launching.
 */
pic_status_t pic_relocate(const pic_geom_t *geom, int32_t batch, int32_t max_docs,
                          int32_t n_pool_docs, const void *k_pool, const void *v_pool,
                          int64_t pool_tokens, const int64_t *doc_token_start,
                          const int32_t *doc_len, const int32_t *doc_base_pos,
                          const int32_t *req_doc_ids, const int32_t *req_num_docs,
                          const int32_t *doc_target, const int32_t *block_table,
                          int32_t max_pages, int64_t num_pages, void *k_cache, void *v_cache,
                          int32_t layer_begin, int32_t layer_end, pic_stream_t stream);

/*
 * pic_relocate_mapped -- pic_relocate driven by pic_compose's token-level
 * maps instead of the per-document description (the same relocation, a
 * CTA per page of logical positions).  For every layer l in [layer_begin,
 * layer_end), request b and position t with tok_map[b][t] = (k << 40) | row:
 *     k_cache[l][slot(t)] = R(doc_delta[b][k]) * k_pool[l][row]
 *     v_cache[l][slot(t)] = v_pool[l][row]                      (bit copy)
 * with slot(t) = slot_mapping[b][t]; arithmetic as pic_relocate, so for the
 * same placement the two give bit-identical caches.
 * Inputs: k_pool, v_pool with pool_tokens rows per layer; tok_map,
 *   slot_mapping int64 [batch][max_ctx]; doc_delta int32 [batch][max_docs].
 * One launch, no workspace.  max_docs == 0 returns PIC_OK without launching.
 */
pic_status_t pic_relocate_mapped(const pic_geom_t *geom, int32_t batch, int32_t max_docs,
                                 const void *k_pool, const void *v_pool, int64_t pool_tokens,
                                 const int64_t *tok_map, const int32_t *doc_delta,
                                 const int64_t *slot_mapping, int32_t max_ctx, int64_t num_pages,
                                 void *k_cache, void *v_cache, int32_t layer_begin,
                                 int32_t layer_end, pic_stream_t stream);

/*
 * pic_link -- pic_compose, pic_relocate_mapped (layers [layer_begin, layer_end)) and
 * pic_append_inline (layer append_layer, or none when append_layer < 0) in a
 * single launch: the link step of a cache hit (Eqs. 1-3; appendix
 * "Position-Independent Linking").  Every argument means what it means for
 * those three calls, and every output -- the layout (doc_offset, doc_delta,
 * slot_mapping, tok_map, inline_pos, ctx_len), the stitched K/V of the
 * documents and of the appended inline tokens, and the packed queries at the
 * start of the prefill workspace -- is bit-identical to theirs (span_len as
 * for pic_compose).  Each CTA handles the positions of one page of one
 * request (two pages when a token's K row has fewer than 1024 elements) for
 * every layer in turn, plus one inline token slot, and derives the layout it
 * needs itself, so the three dependent chains of memory round trips become
 * one.  Requests with more than 256 documents (max_docs > 256) run the three
 * calls in order instead.
 * workspace: the prefill workspace of pic_append_inline (only its leading
 *   packed-query part is written); may be NULL when append_layer < 0.
 * One launch (or the three calls' launches), asynchronous on `stream`;
 * device checks as for the three calls, reported through pic_device_status.
 */
pic_status_t pic_link(const pic_geom_t *geom, int32_t batch, int32_t max_docs,
                      int32_t n_pool_docs, const int32_t *doc_len, const int32_t *doc_base_pos,
                      const int64_t *doc_token_start, const int32_t *req_doc_ids,
                      const int32_t *req_num_docs, const int32_t *span_len,
                      const int32_t *prefix_len, const int32_t *query_len,
                      const int32_t *block_table, int32_t max_pages,
                      int64_t num_pages, int32_t max_ctx, int32_t max_inline, const void *k_pool,
                      const void *v_pool, int64_t pool_tokens, int32_t layer_begin,
                      int32_t layer_end, int32_t append_layer, const void *q, const void *k_new,
                      const void *v_new, const int32_t *inline_len, void *k_cache, void *v_cache,
                      int32_t *doc_offset, int32_t *doc_delta, int64_t *slot_mapping,
                      int64_t *tok_map, int32_t *inline_pos, int32_t *ctx_len, void *workspace,
                      size_t workspace_bytes, pic_stream_t stream);

/*
 * Prefill of one layer's inline tokens ("Cache-hit serving": only the
 * request-specific inline tokens are processed; appendix "Position-Independent
 * Linking": their KVs are interleaved with the prepared document states, and
 * a frontier causal mask stops an inline token from attending to any later
 * logical position).
 *
 * pic_attend_prefill -- given the layer's inline projections q, k_new, v_new
 *   (un-rotated), each inline token t of request b (logical position
 *   p = inline_pos[b][t], t < inline_len[b]) first gets its key R(p) k_new and
 *   value v_new written to slot(p) = block_table[b][p / page] * page + p % page
 *   of `layer` and its query rotated to R(p) q; then for every inline token
 *   and query head h (kv head g = h / G, G = Hq / Hkv):
 *       out[b][t][h] = sum_{s <= p} softmax_s(R(p) q . k_s / sqrt(d)) v_s
 *   over the keys of logical positions 0..p of the stitched cache of `layer`
 *   (the documents relocated there by pic_relocate or pic_link, the inline
 *   tokens just appended).  lse[b][t][h] (nullable) = natural-log sum-exp of
 *   those scaled scores.  Runs on the tensor cores (tcgen05.mma, TMEM
 *   accumulators, TMA loads of the paged K/V through block_table).
 *   num_splits: key-range splits per 128-row query tile (0 = automatic);
 *   splits are merged by log-sum-exp.  Launches: the append, the attention,
 *   the merge when split.
 *   q, k_new, v_new may all be NULL: the append of this layer was already
 *   done into the same workspace by pic_append_inline or pic_link (a fast
 *   path that lets the append overlap other work); the call then only
 *   attends.
 *
 * pic_append_inline -- the append alone (R(p) k_new, v_new into slot(p) =
 *   slot_mapping[b][p], the rotated queries into the workspace, GQA-packed:
 *   the query heads that share a kv head are adjacent rows).  One launch.
 *
 * q: bf16 [batch][max_inline][Hq][d]; k_new, v_new: bf16 [batch][max_inline][Hkv][d]
 *   (un-rotated projections); inline_pos: int32 [batch][max_inline], ascending
 *   per request; inline_len: int32 [batch]; slot_mapping: int64 [batch][max_ctx];
 *   block_table: int32 [batch][max_pages].  Every position must be < max_ctx.
 * out: bf16 [batch][max_inline][Hq][d]; lse: float [batch][max_inline][Hq] or NULL.
 *   out may be page-locked host memory (cudaHostAlloc, cudaHostRegister): the
 *   kernels then store the rows there directly (over the chip-to-chip link of
 *   a Grace-Blackwell node), so a caller that wants the result on the host
 *   needs no copy; PIC_ERR_INVALID_ARG for pageable memory.
 * workspace: >= pic_prefill_workspace_size(... num_splits ...) bytes, 256-byte
 *   aligned (pic_append_inline only uses its leading
 *   pic_prefill_workspace_size(..., 1) bytes).  Device checks: positions in
 *   [0, max_ctx), pages in range, block table long enough.
 */
size_t pic_prefill_workspace_size(const pic_geom_t *geom, int32_t batch, int32_t max_inline,
                                  int32_t max_ctx, int32_t num_splits);

/* Split count pic_attend_prefill uses for these sizes (num_splits 0 = its
 * automatic choice); > 1 means a second (merge) launch.  0 on bad arguments. */
int32_t pic_prefill_num_splits(const pic_geom_t *geom, int32_t batch, int32_t max_inline,
                               int32_t max_ctx, int32_t num_splits);

/* A key-split count for pic_attend_prefill / pic_attend_prefill_fused chosen
 * from the requests' actual inline positions (the logical layout of
 * "Background: Position-Independent Caching" and appendix "Logical Layout
 * and Re-Rotation": prefix, documents, spans, query), which decide how many key tiles
 * each pair of query tiles reads: the call simulates the attention grid's
 * CTAs, in launch order, on the GPU's SMs for every candidate count and
 * returns the one with the least estimated makespan.  Host work only.
 * inline_len: host int32 [batch]; inline_pos: host int32 [batch][max_inline]
 *   (row b's first inline_len[b] entries used), the positions compose writes.
 * Returns 0 on bad arguments (as pic_prefill_num_splits). */
int32_t pic_prefill_plan_splits(const pic_geom_t *geom, int32_t batch, int32_t max_inline,
                                int32_t max_ctx, const int32_t *inline_len,
                                const int32_t *inline_pos);

pic_status_t pic_append_inline(const pic_geom_t *geom, int32_t layer, int32_t batch,
                               int32_t max_inline, const void *q, const void *k_new,
                               const void *v_new, const int32_t *inline_pos,
                               const int32_t *inline_len, const int64_t *slot_mapping,
                               int32_t max_ctx, int64_t num_pages, void *k_cache, void *v_cache,
                               void *workspace, size_t workspace_bytes, pic_stream_t stream);

pic_status_t pic_attend_prefill(const pic_geom_t *geom, int32_t layer, int32_t batch,
                                int32_t max_inline, const void *q, const void *k_new,
                                const void *v_new, const int32_t *inline_pos,
                                const int32_t *inline_len, int32_t max_ctx,
                                const int32_t *block_table, int32_t max_pages, int64_t num_pages,
                                void *k_cache, void *v_cache, void *out, float *lse,
                                int32_t num_splits, void *workspace, size_t workspace_bytes,
                                pic_stream_t stream);

/*
 * pic_attend_prefill_fused -- pic_attend_prefill without the relocated cache:
 * the same outputs, with every document key and value read straight from the
 * pool as it was compiled and the key re-rotation of Eq. 3 applied while the
 * keys are loaded (rotate-on-load), so pic_relocate never runs and the
 * documents' cache slots are never written.
 *
 * Each 128-key tile of the attention is assembled page by page: a page whose
 * 16 positions belong to one document is one box of the document's
 * consecutive pool rows, a page of inline tokens one box of the cache, a page
 * across a boundary is gathered row by row.  The document rows of the key
 * tile are then rotated in shared memory by R(doc_delta[b][k]) with the
 * arithmetic of pic_relocate (fp64-reduced angle, fp32 rotation, bf16 round
 * to nearest even), so the attention reads exactly the keys pic_relocate
 * would have stitched: outputs equal pic_attend_prefill's over that cache
 * bit for bit (same split count).  Values are used as they are.
 *
 * Arguments as pic_attend_prefill, plus: k_pool, v_pool with pool_tokens
 * rows per layer (pool layout above); tok_map int64
 * [batch][max_ctx] and doc_delta int32 [batch][max_docs] as pic_compose (or
 * pic_link) wrote them for this request layout.  Inline keys and values come
 * from the paged cache: pass the layer's projections q, k_new, v_new to
 * append them first, or NULL when pic_append_inline already ran for this
 * layer.  workspace: >= pic_prefill_fused_workspace_size(...) bytes, the
 * same buffer pic_append_inline filled.  Launches: the append when given, a
 * set-up kernel (page sources, document cos/sin), the attention, the merge
 * when split.
 */
/* Workspace of pic_attend_prefill_fused (>= pic_prefill_workspace_size of the
 * same sizes: after the packed queries and split partials, the source of
 * every page of positions < max_ctx and the cos/sin of every listed
 * document).  0 on bad arguments. */
size_t pic_prefill_fused_workspace_size(const pic_geom_t *geom, int32_t batch, int32_t max_inline,
                                        int32_t max_ctx, int32_t max_docs, int32_t num_splits);

pic_status_t pic_attend_prefill_fused(const pic_geom_t *geom, int32_t layer, int32_t batch,
                                      int32_t max_inline, const void *q, const void *k_new,
                                      const void *v_new, const int32_t *inline_pos,
                                      const int32_t *inline_len, int32_t max_ctx,
                                      const int32_t *block_table, int32_t max_pages,
                                      int64_t num_pages, void *k_cache, void *v_cache,
                                      const void *k_pool, const void *v_pool, int64_t pool_tokens,
                                      int32_t max_docs, const int64_t *tok_map,
                                      const int32_t *doc_delta, void *out, float *lse,
                                      int32_t num_splits, void *workspace, size_t workspace_bytes,
                                      pic_stream_t stream);

/*
 * pic_attention_deviation -- the attention-deviation diagnostic of the
 * paper's "Motivating Analysis": D_r(A, B), the mean absolute deviation
 * between the post-softmax attention probabilities of two configurations A
 * and B within normalized block region r.  Here A and B are two stitched key
 * caches of the same requests with the same slot map (for example the
 * relocated cache and one whose documents were copied at their compiled
 * positions), read by the same rotated queries, for one layer.
 * For request b the query rows are its last query_len[b] inline tokens and
 * every query head; the blocks are its documents: token j of document k
 * (n_k tokens) lies in region i when ceil(edges[i] n_k) <= j <
 * ceil(edges[i+1] n_k) (double-precision products), i.e. edges[i] <= j / n_k
 * < edges[i+1].  With p_X = exp(q.k_X / sqrt(d) - lse_X), lse_X the
 * natural-log LSE output of pic_attend_prefill for configuration X:
 *     sums[b][i]   = sum over those rows, heads and keys of |p_A - p_B|
 *     counts[b][i] = the number of terms          (D_i = sums / counts)
 * Inputs (device): inline_pos, inline_len, query_len, req_doc_ids, doc_len,
 *   doc_offset (ascending, -1 past the request's documents), slot_mapping as
 *   from pic_compose / pic_link;
 *   k_cache_a, k_cache_b bf16 paged caches (layout of pic_relocate); lse_a,
 *   lse_b float [batch][max_inline][Hq]; workspace: the prefill workspace
 *   after pic_append_inline (its packed rotated queries are read).
 * edges: HOST array of n_regions + 1 ascending fractions in [0, 1],
 *   1 <= n_regions <= 8 (e.g. {0, 0.1, 0.9}: the paper's pre and int regions).
 * max_query_len: the largest query_len[b] (host value; sizes the grid).
 * Outputs (device, overwritten): sums double [batch][n_regions], counts
 *   int64 [batch][n_regions].  Two memsets and one launch on `stream`: a
 *   tcgen05 kernel (both score matrices on the tensor cores; a diagnostic,
 *   off the serving path).  Each CTA keeps its request's document table in
 *   shared memory: PIC_ERR_UNSUPPORTED when max_docs x 4 (n_regions + 3)
 *   bytes do not fit beside the tiles (about 60 KB: 1500-3000 documents).
 */
pic_status_t pic_attention_deviation(const pic_geom_t *geom, int32_t layer, int32_t batch,
                                     int32_t max_inline, int32_t max_docs, int32_t max_ctx,
                                     int64_t num_pages, const int32_t *inline_pos,
                                     const int32_t *inline_len, const int32_t *query_len,
                                     int32_t max_query_len, const int32_t *req_doc_ids,
                                     const int32_t *doc_len,
                                     const int32_t *doc_offset, const int64_t *slot_mapping,
                                     const void *k_cache_a,
                                     const void *k_cache_b, const float *lse_a,
                                     const float *lse_b, const double *edges, int32_t n_regions,
                                     const void *workspace, size_t workspace_bytes, double *sums,
                                     int64_t *counts, pic_stream_t stream);

/*
 * pic_attend_decode -- one layer of one plain autoregressive decoding step over
 * the completed cache (appendix "Position-Independent Linking": after the first
 * token, generation proceeds as usual on the linked cache).
 *
 * For each request b with new-token position p = pos[b] + pos_offset:
 *   k_cache/v_cache[layer][slot(p)] = R(p) k_new[b], v_new[b];
 *   out[b][h] = sum_{s <= p} softmax_s(R(p) q[b][h] . k_s / sqrt(d)) v_s.
 * slot(p) = block_table[b][p / page] * page + p % page.
 * q: bf16 [batch][Hq][d]; k_new, v_new: bf16 [batch][Hkv][d]; pos: int32 [batch]
 * (e.g. ctx_len from pic_compose) plus the scalar pos_offset (e.g. the step index);
 * out: bf16 [batch][Hq][d]; lse: float [batch][Hq] or NULL.
 * max_ctx: an upper bound on pos[b] + pos_offset + 1 (sizes the grid); a
 * request whose keys reach past it is reported as PIC_DEV_CTX_OVERFLOW by
 * pic_device_status (its output then misses those keys).
 * num_splits: key-range splits per (request, kv head) (0 = automatic); the
 * partial softmax states are merged by log-sum-exp.  Hq / Hkv <= 16.
 * workspace: >= pic_decode_workspace_size(... same num_splits ...) bytes.
 */
size_t pic_decode_workspace_size(const pic_geom_t *geom, int32_t batch, int32_t max_ctx,
                                 int32_t num_splits);

/* Split count pic_attend_decode uses for these sizes (0 on bad arguments). */
int32_t pic_decode_num_splits(const pic_geom_t *geom, int32_t batch, int32_t max_ctx,
                              int32_t num_splits);

pic_status_t pic_attend_decode(const pic_geom_t *geom, int32_t layer, int32_t batch,
                               const void *q, const void *k_new, const void *v_new,
                               const int32_t *pos, int32_t pos_offset, const int32_t *block_table,
                               int32_t max_pages, int64_t num_pages, void *k_cache,
                               void *v_cache, void *out, float *lse, int32_t max_ctx,
                               int32_t num_splits, void *workspace, size_t workspace_bytes,
                               pic_stream_t stream);

/*
 * pic_attend_decode_noalloc -- pic_attend_decode for callers that cannot
 * allocate device memory while they decode (an engine that gave its whole
 * memory budget to the KV cache, a runtime that forbids allocation after
 * start-up, a plugin that only owns the tensors it is handed).  The paper has
 * no counterpart: this is a deployment convenience of this library.
 *
 * Same arguments and results as pic_attend_decode, without the workspace:
 * the scratch (rotated queries, per-split partial softmax states) lives in an
 * 8 MiB array inside the library that every GPU which loads it holds until
 * the process exits.  The call allocates nothing.
 *  - The first call on a device (with that device current) looks the array
 *    up with cudaGetSymbolAddress (and again after a device reset, which
 *    gives the device a new context); make that first call before any
 *    stream capture.
 *  - Every call on a device shares the array: calls that overlap on the GPU
 *    (e.g. on two streams) race.  No scratch value needs to start at zero.
 *  - num_splits 0 picks the automatic split count, lowered until the scratch
 *    fits; an explicit num_splits whose scratch exceeds 8 MiB, or a problem
 *    too large even with one split, returns PIC_ERR_WORKSPACE.
 */
pic_status_t pic_attend_decode_noalloc(const pic_geom_t *geom, int32_t layer, int32_t batch,
                                       const void *q, const void *k_new, const void *v_new,
                                       const int32_t *pos, int32_t pos_offset,
                                       const int32_t *block_table, int32_t max_pages,
                                       int64_t num_pages, void *k_cache, void *v_cache, void *out,
                                       float *lse, int32_t max_ctx, int32_t num_splits,
                                       pic_stream_t stream);

#ifdef __cplusplus
} /* extern "C" */
#endif

#endif /* PIC_H_ */
