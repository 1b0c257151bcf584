// pic_relocate: key re-rotation (Eq. 3) and stitching of cached documents
// into the paged request cache; values are copied unchanged (the paper rotates
// keys only; Background: Position-Independent Caching).
//
// One launch, one CTA per (one or two pages of logical positions, request);
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
};

// kLayerRope: a rotary table per layer (its cos/sin double-buffered: the next
// layer's table is computed while this layer's loads are in flight)
template <int D, int kTok, bool kLayerRope>
__global__ void __launch_bounds__(kThreads) relocate_kernel(RelocArgs a, RopeParams rp) {
  static_assert(kTok == 16 || kTok == 32, "one warp scans the positions of a CTA");
  pdl_entry();
  constexpr unsigned kMask = kTok == 32 ? 0xffffffffu : 0x0000ffffu;
  constexpr int HALF = D / 2;
  constexpr int KC = D / 16;  // 8-pair chunks per K row
  constexpr int VC = D / 8;   // 16-byte pieces per V row
  const int style = rp.style;
  const int b = blockIdx.y;
  const long long t0 = (long long)blockIdx.x * kTok;
  const int tid = threadIdx.x;

  __shared__ long long s_src[kTok];  // pool row of position t0 + i, -1 = not a doc token
  __shared__ long long s_dst[kTok];  // cache slot
  __shared__ int s_doc[kTok];        // document index k within the request
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

  const size_t hkv = a.hkv;
  auto fill_cs = [&](int layer, int buf) {  // cos/sin of the touched documents
    for (int e = tid; e < n_docs * HALF; e += kThreads) {
      const int j = e / HALF, i = e % HALF;
      const int delta = a.delta[(size_t)b * a.max_docs + k_first + j];
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

extern "C" pic_status_t pic_relocate(const pic_geom_t *geom, int32_t batch, int32_t max_docs,
                                     const void *k_pool, const void *v_pool, int64_t pool_tokens,
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
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: sizes must be positive");
  if (pool_tokens >= (1LL << 40))
    return fail(PIC_ERR_UNSUPPORTED, "pic_relocate: pool has 2^40 rows or more");
  if (layer_begin < 0 || layer_end > geom->num_layers || layer_begin >= layer_end)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: layer range [%d, %d) outside [0, %d)",
                layer_begin, layer_end, geom->num_layers);
  if (layer_end - layer_begin > 65535 || batch > 65535)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: grid too large");
  if (!k_pool || !v_pool || !tok_map || !doc_delta || !slot_mapping || !k_cache || !v_cache)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: NULL tensor");
  if ((reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
       reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: K/V tensors must be 16-byte aligned");
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_relocate: no device status word");

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
  if (e != cudaSuccess) return cuda_fail(e, "pic_relocate launch");
  return PIC_OK;
}
