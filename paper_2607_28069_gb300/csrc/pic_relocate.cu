// pic_relocate / pic_relocate_mapped: key re-rotation (Eq. 3) and stitching
// of cached documents into the paged request cache; values are copied
// unchanged (the paper rotates keys only; Background: Position-Independent
// Caching).
//
// pic_relocate takes the problem as the paper states it: per listed document
// its pool rows, base position and target position, and the request's block
// table (relocate_docs_kernel: a CTA per chunk of a document's tokens).
// pic_relocate_mapped takes pic_compose's token and slot maps instead
// (relocate_kernel, described below); both share the mover of the second
// half, so for the same placement their caches are bit-identical.
//
// relocate_kernel: one launch, one CTA per (one or two pages of logical
// positions, request);
// the CTA moves its positions for every layer in turn, so its set-up (maps,
// cos/sin) is done once and it keeps a long stream of loads in flight.
// The CTA reads the token map and slot map of its positions (written by
// pic_compose) and evaluates cos/sin of delta_k * theta_i for the documents
// its page touches; then, per layer, it issues every K and V load of its page
// at once (16-byte streaming loads; V rows are bit copies, K rows come as the
// two 16-byte halves of 8 RoPE pairs), rotates and stores.  delta is
// constant over a document because base and target positions both advance by
// one per token, so R(b) R(a)^-1 = R(b - a) = R(delta).  The angle is formed and
// reduced in fp64, sin/cos evaluated in fp32 on the reduced angle; K is rotated
// in fp32 and rounded to bf16 (round to nearest even).  Pool rows and cache
// rows are d contiguous bf16 and consecutive threads take consecutive 16-byte
// pieces of the same row, so every warp access is fully coalesced.
// HBM-bound: 4 * Hkv * d * 2 bytes move per document token.
#include <algorithm>

#include "pic_internal.cuh"

namespace pic {
namespace {

constexpr int kThreads = 256;
// Positions per CTA: one page (16) when a token carries >= 1024 K elements,
// two pages otherwise, so every CTA moves 64 KB and amortises its set-up.
constexpr int UV = 8;     // V tasks per thread per round
constexpr int UK = 4;     // K tasks per thread per round

struct RelocArgs {
  int max_docs, max_ctx, hkv, layer_begin, layer_end;
  long long pool_tokens, num_pages;
  const __nv_bfloat16 *k_pool, *v_pool;
  const int64_t *tok_map, *slots;
  const int32_t *delta;
  __nv_bfloat16 *k_cache, *v_cache;
  int32_t *status;
  // per-document form (pic_relocate): the documents' pool rows, base and
  // target positions, and the block table instead of the two maps
  int n_pool_docs, max_pages;
  const int64_t *doc_start;
  const int32_t *doc_len, *doc_base, *ids, *num_docs, *target, *block_table;
};

// Moves the positions a CTA set up (s_src / s_dst / s_doc, the documents'
// deltas in s_delta) for every layer of [layer_begin, layer_end): the
// shared second half of both relocation kernels.
template <int D, int kTok, bool kLayerRope>
__device__ __forceinline__ void move_positions(const RelocArgs &a, const RopeParams &rp, int b,
                                               const long long *s_src, const long long *s_dst,
                                               const int *s_doc, const int *s_delta,
                                               int k_first, int n_docs,
                                               float2 (*s_cs)[kTok][D / 2]);

// kLayerRope: a rotary table per layer (its cos/sin double-buffered: the next
// layer's table is computed while this layer's loads are in flight)
template <int D, int kTok, bool kLayerRope>
__global__ void __launch_bounds__(kThreads) relocate_kernel(RelocArgs a, RopeParams rp) {
  static_assert(kTok == 16 || kTok == 32, "one warp scans the positions of a CTA");
  pdl_entry();
  constexpr unsigned kMask = kTok == 32 ? 0xffffffffu : 0x0000ffffu;
  constexpr int HALF = D / 2;
  const int b = blockIdx.y;
  const long long t0 = (long long)blockIdx.x * kTok;
  const int tid = threadIdx.x;

  __shared__ long long s_src[kTok];  // pool row of position t0 + i, -1 = not a doc token
  __shared__ long long s_dst[kTok];  // cache slot
  __shared__ int s_doc[kTok];        // document index k within the request
  __shared__ int s_delta[kTok];      // delta of documents k_first .. k_first + n_docs - 1
  __shared__ int s_first, s_last;    // document range touched by this page
  __shared__ float2 s_cs[kLayerRope ? 2 : 1][kTok][HALF];

  if (tid < kTok) {
    const long long t = t0 + tid;
    long long src = -1, slot = -1;
    int k = 0;
    if (t < a.max_ctx) {
      const long long tm = a.tok_map[(size_t)b * a.max_ctx + t];
      slot = a.slots[(size_t)b * a.max_ctx + t];
      if (tm >= 0) {
        k = (int)(tm >> 40);
        src = tm & ((1LL << 40) - 1);
        if (src >= a.pool_tokens || k >= a.max_docs) {
          dev_fail(a.status, PIC_DEV_BAD_DOC_LEN, b);
          src = -1;
        } else if (slot < 0 || slot >= a.num_pages * 16) {
          dev_fail(a.status, PIC_DEV_BAD_PAGE, b);
          src = -1;
        }
      }
    }
    s_src[tid] = src;
    s_dst[tid] = slot;
    s_doc[tid] = k;
    // documents of a page are consecutive: first / last valid position's doc
    const unsigned valid = __ballot_sync(kMask, src >= 0);
    const int kf = __shfl_sync(kMask, k, valid ? __ffs(valid) - 1 : 0);
    const int kl = __shfl_sync(kMask, k, valid ? 31 - __clz(valid) : 0);
    if (tid == 0) {
      s_first = valid ? kf : -1;
      s_last = valid ? kl : -1;
    }
  }
  __syncthreads();
  if (s_first < 0) return;  // no document token on this page
  const int k_first = s_first;
  // every document between the first and last one here owns >= 1 position,
  // so at most kTok rows; anything else is a malformed token map
  const int n_docs = min(s_last - s_first + 1, kTok);
  if (tid < n_docs) s_delta[tid] = a.delta[(size_t)b * a.max_docs + k_first + tid];
  __syncthreads();
  move_positions<D, kTok, kLayerRope>(a, rp, b, s_src, s_dst, s_doc, s_delta, k_first, n_docs,
                                      s_cs);
}

// The per-document form: CTA (slice, k, b) moves the kTok-token chunks
// slice, slice + S, ... of the k-th listed document of request b (S =
// gridDim.x): token j of the document (pool row doc_start + j, compiled at
// base + j) goes to logical position target + j, i.e. to slot
// block_table[b][(target + j) / 16] * 16 + (target + j) % 16, rotated by
// delta = target - base.
template <int D, int kTok, bool kLayerRope>
__global__ void __launch_bounds__(kThreads) relocate_docs_kernel(RelocArgs a, RopeParams rp) {
  pdl_entry();
  constexpr int HALF = D / 2;
  const int k = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  __shared__ long long s_src[kTok];
  __shared__ long long s_dst[kTok];
  __shared__ int s_doc[kTok];
  __shared__ int s_delta[1];
  __shared__ float2 s_cs[kLayerRope ? 2 : 1][kTok][HALF];
  const int m = a.num_docs[b];
  if (m < 0 || m > a.max_docs) {
    if (tid == 0 && blockIdx.x == 0 && k == 0) dev_fail(a.status, PIC_DEV_BAD_REQUEST, b);
    return;
  }
  if (k >= m) return;
  const int id = a.ids[(size_t)b * a.max_docs + k];
  if (id < 0 || id >= a.n_pool_docs) {
    if (tid == 0 && blockIdx.x == 0) dev_fail(a.status, PIC_DEV_BAD_DOC_ID, b);
    return;
  }
  const int n = a.doc_len[id];
  const long long start = a.doc_start[id];
  if (n <= 0 || start < 0 || start + n > a.pool_tokens) {
    if (tid == 0 && blockIdx.x == 0) dev_fail(a.status, PIC_DEV_BAD_DOC_LEN, b);
    return;
  }
  const long long target = a.target[(size_t)b * a.max_docs + k];
  if (target < 0 || target + n > (long long)a.max_pages * 16) {
    if (tid == 0 && blockIdx.x == 0)
      dev_fail(a.status, target < 0 ? PIC_DEV_BAD_POSITION : PIC_DEV_BLOCK_TABLE_SHORT, b);
    return;
  }
  if (blockIdx.x == 0 && tid < 32) {  // targets of two listed documents must not overlap
    bool clash = false;
    for (int k2 = tid; k2 < m; k2 += 32) {
      if (k2 == k) continue;
      const int id2 = a.ids[(size_t)b * a.max_docs + k2];
      if (id2 < 0 || id2 >= a.n_pool_docs) continue;
      const long long t2 = a.target[(size_t)b * a.max_docs + k2];
      const long long n2 = a.doc_len[id2];
      clash |= t2 < target + n && target < t2 + n2;
    }
    if (__any_sync(0xffffffffu, clash) && tid == 0) dev_fail(a.status, PIC_DEV_BAD_POSITION, b);
  }
  if (tid == 0) s_delta[0] = (int)(target - a.doc_base[id]);
  const int32_t *bt = a.block_table + (size_t)b * a.max_pages;
  const int chunks = (n + kTok - 1) / kTok;
  for (int c = blockIdx.x; c < chunks; c += gridDim.x) {
    __syncthreads();  // the previous chunk's maps are no longer read
    if (tid < kTok) {
      const int j = c * kTok + tid;
      long long src = -1, slot = -1;
      if (j < n) {
        const long long t = target + j;
        const int page = bt[t >> 4];
        if (page < 0 || page >= a.num_pages) {
          dev_fail(a.status, PIC_DEV_BAD_PAGE, b);
        } else {
          src = start + j;
          slot = (long long)page * 16 + (t & 15);
        }
      }
      s_src[tid] = src;
      s_dst[tid] = slot;
      s_doc[tid] = 0;
    }
    __syncthreads();
    move_positions<D, kTok, kLayerRope>(a, rp, b, s_src, s_dst, s_doc, s_delta, 0, 1, s_cs);
  }
}

template <int D, int kTok, bool kLayerRope>
__device__ __forceinline__ void move_positions(const RelocArgs &a, const RopeParams &rp, int b,
                                               const long long *s_src, const long long *s_dst,
                                               const int *s_doc, const int *s_delta,
                                               int k_first, int n_docs,
                                               float2 (*s_cs)[kTok][D / 2]) {
  constexpr int HALF = D / 2;
  constexpr int KC = D / 16;  // 8-pair chunks per K row
  constexpr int VC = D / 8;   // 16-byte pieces per V row
  const int style = rp.style;
  const int tid = threadIdx.x;
  const size_t hkv = a.hkv;
  auto fill_cs = [&](int layer, int buf) {  // cos/sin of the touched documents
    for (int e = tid; e < n_docs * HALF; e += kThreads) {
      const int j = e / HALF, i = e % HALF;
      const int delta = s_delta[j];
      s_cs[buf][j][i] = kLayerRope ? rope_cos_sin_fast(delta, rope_theta(rp, layer, i))
                                   : rope_cos_sin(delta, rope_theta(rp, layer, i));
    }
  };
  fill_cs(a.layer_begin, 0);
  __syncthreads();
  for (int layer = a.layer_begin; layer < a.layer_end; ++layer) {
  const int cur = kLayerRope ? (layer - a.layer_begin) & 1 : 0;
  const __nv_bfloat16 *kp = a.k_pool + (size_t)layer * a.pool_tokens * hkv * D;
  const __nv_bfloat16 *vp = a.v_pool + (size_t)layer * a.pool_tokens * hkv * D;
  __nv_bfloat16 *kc = a.k_cache + (size_t)layer * a.num_pages * hkv * 16 * D;
  __nv_bfloat16 *vc = a.v_cache + (size_t)layer * a.num_pages * hkv * 16 * D;
  const int nV = kTok * (int)hkv * VC, nK = kTok * (int)hkv * KC;

  for (int round = 0; round * kThreads * UV < nV || round * kThreads * UK < nK; ++round) {
    // ---- issue this round's loads
    uint4 v[UV], ka[UK], kb[UK];
    long long vdst[UV], kdst[UK];
    int kdoc[UK], kch[UK];
#pragma unroll
    for (int u = 0; u < UV; ++u) {
      const int task = (round * UV + u) * kThreads + tid;
      vdst[u] = -1;
      if (task < nV) {
        const int i = task / ((int)hkv * VC), r = task % ((int)hkv * VC);
        const int h = r / VC, c = r % VC;
        const long long src = s_src[i];
        if (src >= 0) {
          const long long slot = s_dst[i];
          v[u] = ld_stream(vp + ((size_t)src * hkv + h) * D + c * 8);
          vdst[u] = (((slot >> 4) * (long long)hkv + h) * 16 + (slot & 15)) * D + c * 8;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < UK; ++u) {
      const int task = (round * UK + u) * kThreads + tid;
      kdst[u] = -1;
      if (task < nK) {
        const int i = task / ((int)hkv * KC), r = task % ((int)hkv * KC);
        const int h = r / KC, c = r % KC;
        const long long src = s_src[i];
        if (src >= 0) {
          const long long slot = s_dst[i];
          const PairChunk pc = pair_chunk(c, HALF, style);
          const __nv_bfloat16 *sp = kp + ((size_t)src * hkv + h) * D;
          ka[u] = ld_stream(sp + pc.off_a);
          kb[u] = ld_stream(sp + pc.off_b);
          kdst[u] = (((slot >> 4) * (long long)hkv + h) * 16 + (slot & 15)) * D;
          kdoc[u] = s_doc[i] - k_first;
          kch[u] = c;
          if (kdoc[u] >= n_docs) kdst[u] = -1;
        }
      }
    }
    if constexpr (kLayerRope) {  // next layer's table while the loads are in flight
      if (round == 0 && layer + 1 < a.layer_end) fill_cs(layer + 1, cur ^ 1);
    }
    // ---- V: bit copy
#pragma unroll
    for (int u = 0; u < UV; ++u)
      if (vdst[u] >= 0) st_global16(vc + vdst[u], v[u]);
    // ---- K: rotate 8 pairs and store
#pragma unroll
    for (int u = 0; u < UK; ++u) {
      if (kdst[u] < 0) continue;
      const int c = kch[u];
      float2 cs[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) cs[q] = s_cs[cur][kdoc[u]][8 * c + q];
      float x[8], y[8], uu[8], ww[8];
      unpack8(ka[u], x);
      unpack8(kb[u], y);
      if (style == PIC_ROPE_HALF) {
#pragma unroll
        for (int q = 0; q < 8; ++q) { uu[q] = x[q]; ww[q] = y[q]; }
      } else {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uu[q] = x[2 * q]; ww[q] = x[2 * q + 1];
          uu[4 + q] = y[2 * q]; ww[4 + q] = y[2 * q + 1];
        }
      }
      rotate8(uu, ww, cs);
      if (style == PIC_ROPE_HALF) {
#pragma unroll
        for (int q = 0; q < 8; ++q) { x[q] = uu[q]; y[q] = ww[q]; }
      } else {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          x[2 * q] = uu[q]; x[2 * q + 1] = ww[q];
          y[2 * q] = uu[4 + q]; y[2 * q + 1] = ww[4 + q];
        }
      }
      const PairChunk pc = pair_chunk(c, HALF, style);
      st_global16(kc + kdst[u] + pc.off_a, pack8(x));
      st_global16(kc + kdst[u] + pc.off_b, pack8(y));
    }
  }
  if constexpr (kLayerRope) __syncthreads();  // next table written; this one read
  }
}

}  // namespace
}  // namespace pic

extern "C" pic_status_t pic_relocate_mapped(const pic_geom_t *geom, int32_t batch,
                                            int32_t max_docs, const void *k_pool,
                                            const void *v_pool, int64_t pool_tokens,
                                            const int64_t *tok_map, const int32_t *doc_delta,
                                            const int64_t *slot_mapping, int32_t max_ctx,
                                            int64_t num_pages, void *k_cache, void *v_cache,
                                            int32_t layer_begin, int32_t layer_end,
                                            pic_stream_t stream) {
  using namespace pic;
  RopeParams rp;
  pic_status_t st = make_rope(geom, &rp);
  if (st != PIC_OK) return st;
  if (max_docs == 0 && batch > 0) return PIC_OK;  // no document to move
  if (batch <= 0 || max_docs < 0 || pool_tokens <= 0 || max_ctx <= 0 || num_pages <= 0)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate_mapped: sizes must be positive");
  if (pool_tokens >= (1LL << 40))
    return fail(PIC_ERR_UNSUPPORTED, "pic_relocate_mapped: pool has 2^40 rows or more");
  if (layer_begin < 0 || layer_end > geom->num_layers || layer_begin >= layer_end)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate_mapped: layer range [%d, %d) outside [0, %d)",
                layer_begin, layer_end, geom->num_layers);
  if (layer_end - layer_begin > 65535 || batch > 65535)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate_mapped: grid too large");
  if (!k_pool || !v_pool || !tok_map || !doc_delta || !slot_mapping || !k_cache || !v_cache)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate_mapped: NULL tensor");
  if ((reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
       reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate_mapped: K/V tensors must be 16-byte aligned");
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_relocate_mapped: no device status word");

  RelocArgs a;
  a.max_docs = max_docs;
  a.max_ctx = max_ctx;
  a.hkv = geom->num_kv_heads;
  a.layer_begin = layer_begin;
  a.layer_end = layer_end;
  a.pool_tokens = pool_tokens;
  a.num_pages = num_pages;
  a.k_pool = static_cast<const __nv_bfloat16 *>(k_pool);
  a.v_pool = static_cast<const __nv_bfloat16 *>(v_pool);
  a.tok_map = tok_map;
  a.slots = slot_mapping;
  a.delta = doc_delta;
  a.k_cache = static_cast<__nv_bfloat16 *>(k_cache);
  a.v_cache = static_cast<__nv_bfloat16 *>(v_cache);
  a.status = status;
  const bool wide = geom->num_kv_heads * geom->head_dim >= 1024;
  const int tok = wide ? 16 : 32;
  dim3 grid((max_ctx + tok - 1) / tok, batch);
  const dim3 block(kThreads);
  cudaError_t e;
  if (geom->head_dim == 128)
    e = rp.layer_theta
            ? (wide ? launch_dependent(relocate_kernel<128, 16, true>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_kernel<128, 32, true>, grid, block, 0, stream, a, rp))
            : (wide ? launch_dependent(relocate_kernel<128, 16, false>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_kernel<128, 32, false>, grid, block, 0, stream, a, rp));
  else
    e = rp.layer_theta
            ? (wide ? launch_dependent(relocate_kernel<64, 16, true>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_kernel<64, 32, true>, grid, block, 0, stream, a, rp))
            : (wide ? launch_dependent(relocate_kernel<64, 16, false>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_kernel<64, 32, false>, grid, block, 0, stream, a, rp));
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_relocate_mapped launch");
  return PIC_OK;
}

extern "C" pic_status_t pic_relocate(const pic_geom_t *geom, int32_t batch, int32_t max_docs,
                                     int32_t n_pool_docs, const void *k_pool, const void *v_pool,
                                     int64_t pool_tokens, const int64_t *doc_token_start,
                                     const int32_t *doc_len, const int32_t *doc_base_pos,
                                     const int32_t *req_doc_ids, const int32_t *req_num_docs,
                                     const int32_t *doc_target, const int32_t *block_table,
                                     int32_t max_pages, int64_t num_pages, void *k_cache,
                                     void *v_cache, int32_t layer_begin, int32_t layer_end,
                                     pic_stream_t stream) {
  using namespace pic;
  RopeParams rp;
  pic_status_t st = make_rope(geom, &rp);
  if (st != PIC_OK) return st;
  if (max_docs == 0 && batch > 0) return PIC_OK;  // no document to move
  if (batch <= 0 || max_docs < 0 || n_pool_docs <= 0 || pool_tokens <= 0 || max_pages <= 0 ||
      num_pages <= 0)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: sizes must be positive");
  if (layer_begin < 0 || layer_end > geom->num_layers || layer_begin >= layer_end)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: layer range [%d, %d) outside [0, %d)",
                layer_begin, layer_end, geom->num_layers);
  if (max_docs > 65535 || batch > 65535)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: grid too large");
  if ((long long)max_pages * 16 >= (1LL << 31))
    return fail(PIC_ERR_UNSUPPORTED, "pic_relocate: block table longer than 2^27 pages");
  if (!k_pool || !v_pool || !doc_token_start || !doc_len || !doc_base_pos || !req_doc_ids ||
      !req_num_docs || !doc_target || !block_table || !k_cache || !v_cache)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: NULL tensor");
  if ((reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
       reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: K/V tensors must be 16-byte aligned");
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_relocate: no device status word");

  RelocArgs a = {};
  a.max_docs = max_docs;
  a.hkv = geom->num_kv_heads;
  a.layer_begin = layer_begin;
  a.layer_end = layer_end;
  a.pool_tokens = pool_tokens;
  a.num_pages = num_pages;
  a.k_pool = static_cast<const __nv_bfloat16 *>(k_pool);
  a.v_pool = static_cast<const __nv_bfloat16 *>(v_pool);
  a.k_cache = static_cast<__nv_bfloat16 *>(k_cache);
  a.v_cache = static_cast<__nv_bfloat16 *>(v_cache);
  a.status = status;
  a.n_pool_docs = n_pool_docs;
  a.max_pages = max_pages;
  a.doc_start = doc_token_start;
  a.doc_len = doc_len;
  a.doc_base = doc_base_pos;
  a.ids = req_doc_ids;
  a.num_docs = req_num_docs;
  a.target = doc_target;
  a.block_table = block_table;
  const bool wide = geom->num_kv_heads * geom->head_dim >= 1024;
  // slices per document: each CTA walks every slices-th chunk of its document;
  // few documents get more slices (up to one chunk per CTA), so that a small
  // request still fills the GPU (CTAs past a document's last chunk exit)
  const long long docs_total = (long long)batch * max_docs;
  const int slices = (int)std::min<long long>(128, std::max<long long>(16, (8 * 152 + docs_total - 1) / docs_total));
  dim3 grid(slices, max_docs, batch);
  const dim3 block(kThreads);
  cudaError_t e;
  if (geom->head_dim == 128)
    e = rp.layer_theta
            ? (wide ? launch_dependent(relocate_docs_kernel<128, 16, true>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_docs_kernel<128, 32, true>, grid, block, 0, stream, a, rp))
            : (wide ? launch_dependent(relocate_docs_kernel<128, 16, false>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_docs_kernel<128, 32, false>, grid, block, 0, stream, a, rp));
  else
    e = rp.layer_theta
            ? (wide ? launch_dependent(relocate_docs_kernel<64, 16, true>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_docs_kernel<64, 32, true>, grid, block, 0, stream, a, rp))
            : (wide ? launch_dependent(relocate_docs_kernel<64, 16, false>, grid, block, 0, stream, a, rp)
                    : launch_dependent(relocate_docs_kernel<64, 32, false>, grid, block, 0, stream, a, rp));
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_relocate launch");
  return PIC_OK;
}
