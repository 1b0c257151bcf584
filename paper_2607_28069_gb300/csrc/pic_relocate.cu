// pic_relocate: key re-rotation (Eq. 3) and stitching of cached documents
// into the paged request cache; values are copied unchanged (the paper rotates
// keys only; Background: Position-Independent Caching).
//
// One launch, one CTA per (16 logical positions = one page, request, layer).
// The CTA finds which documents overlap its positions, copies the V rows (bit
// copy), evaluates cos/sin of delta_k * theta_i for the documents it touches
// (delta is constant over a document because base and target positions both
// advance by one per token, so R(b) R(a)^-1 = R(b - a) = R(delta); the angle is
// formed and reduced in fp64, sin/cos evaluated in fp32 on the reduced angle),
// then rotates the K rows in fp32 and rounds them to bf16 (round to nearest
// even).  Pool rows and cache rows are both d contiguous bf16 and consecutive
// threads take consecutive 16-byte pieces of the same row, so every warp
// access is fully coalesced.  HBM-bound: 4 * Hkv * d * 2 bytes move per token.
#include "pic_internal.cuh"

namespace pic {
namespace {

constexpr int kThreads = 256;
constexpr int kTok = 16;  // positions per CTA (one page)

struct RelocArgs {
  int max_docs, n_pool, max_ctx, hkv, layer_begin;
  long long pool_tokens, num_pages;
  const __nv_bfloat16 *k_pool, *v_pool;
  const int64_t *doc_start;
  const int32_t *doc_len, *ids, *num_docs, *offset;
  const int32_t *delta;
  const int64_t *slots;
  __nv_bfloat16 *k_cache, *v_cache;
  int32_t *status;
};

template <int D>
__global__ void __launch_bounds__(kThreads) relocate_kernel(RelocArgs a, RopeParams rp) {
  const int style = rp.style;
  constexpr int HALF = D / 2;
  constexpr int KC = D / 16;  // 8-pair chunks per K row
  constexpr int VC = D / 8;   // 16-byte pieces per V row
  const int b = blockIdx.y;
  const int layer = a.layer_begin + blockIdx.z;
  const long long t0 = (long long)blockIdx.x * kTok;
  const int tid = threadIdx.x;

  __shared__ long long s_src[kTok];  // pool row of position t0 + i, -1 = not a doc token
  __shared__ long long s_dst[kTok];  // cache slot
  __shared__ int s_tab[kTok];        // row of s_cs used by position t0 + i
  __shared__ int s_doc[kTok];        // documents touching this page (k index)
  __shared__ int s_ndoc;
  __shared__ float2 s_cs[kTok][HALF];  // cos/sin of delta_k * theta_i per touching doc
  if (tid < kTok) s_src[tid] = -1;
  if (tid == 0) s_ndoc = 0;
  __syncthreads();

  const int m = a.num_docs[b];
  if (m <= 0 || m > a.max_docs) return;
  const int32_t *off = a.offset + (size_t)b * a.max_docs;
  const int32_t *ids = a.ids + (size_t)b * a.max_docs;
  for (int k = tid; k < m; k += kThreads) {
    const long long o = off[k];
    if (o >= t0 + kTok || o < 0) continue;
    const int id = ids[k];
    if (id < 0 || id >= a.n_pool) continue;  // reported by pic_compose
    const long long n = a.doc_len[id];
    if (o + n <= t0) continue;
    const long long start = a.doc_start[id];
    if (n <= 0 || start < 0 || start + n > a.pool_tokens) {
      dev_fail(a.status, PIC_DEV_BAD_DOC_LEN, b);
      continue;
    }
    const int slot_of_doc = atomicAdd(&s_ndoc, 1);  // < kTok: each doc owns >= 1 position here
    s_doc[slot_of_doc] = k;
    for (long long t = max(o, t0); t < min(o + n, t0 + kTok); ++t) {
      const int i = (int)(t - t0);
      long long slot = t < a.max_ctx ? a.slots[(size_t)b * a.max_ctx + t] : -1;
      if (slot < 0 || slot >= a.num_pages * 16) {
        dev_fail(a.status, PIC_DEV_BAD_PAGE, b);
        continue;
      }
      s_src[i] = start + (t - o);
      s_dst[i] = slot;
      s_tab[i] = slot_of_doc;
    }
  }
  __syncthreads();

  const size_t hkv = a.hkv;
  const __nv_bfloat16 *kp = a.k_pool + (size_t)layer * a.pool_tokens * hkv * D;
  const __nv_bfloat16 *vp = a.v_pool + (size_t)layer * a.pool_tokens * hkv * D;
  __nv_bfloat16 *kc = a.k_cache + (size_t)layer * a.num_pages * hkv * 16 * D;
  __nv_bfloat16 *vc = a.v_cache + (size_t)layer * a.num_pages * hkv * 16 * D;

  // V: bit copy, 8 independent 16-byte loads in flight per thread.
  {
    constexpr int U = 8;
    const int total = kTok * (int)hkv * VC;
    for (int base = tid; base < total; base += kThreads * U) {
      uint4 v[U];
      long long dst[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int task = base + u * kThreads;
        dst[u] = -1;
        if (task < total) {
          const int i = task / ((int)hkv * VC), r = task % ((int)hkv * VC);
          const int h = r / VC, c = r % VC;
          const long long src = s_src[i];
          if (src >= 0) {
            const long long slot = s_dst[i];
            v[u] = ld_stream(vp + ((size_t)src * hkv + h) * D + c * 8);
            dst[u] = (((slot >> 4) * (long long)hkv + h) * 16 + (slot & 15)) * D + c * 8;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (dst[u] >= 0) st_global16(vc + dst[u], v[u]);
    }
  }
  // cos/sin of the documents touching this page (issued after the V loads)
  for (int e = tid; e < s_ndoc * HALF; e += kThreads) {
    const int j = e / HALF, i = e % HALF;
    const int delta = a.delta[(size_t)b * a.max_docs + s_doc[j]];
    s_cs[j][i] = rope_cos_sin(delta, rp.theta[i]);
  }
  __syncthreads();
  // K: rotate 8 pairs per task (two 16-byte pieces), 4 tasks in flight.
  {
    constexpr int U = 4;
    const int total = kTok * (int)hkv * KC;
    for (int base = tid; base < total; base += kThreads * U) {
      uint4 va[U], vb[U];
      long long dst[U];
      int tab[U], chunk[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int task = base + u * kThreads;
        dst[u] = -1;
        if (task < total) {
          const int i = task / ((int)hkv * KC), r = task % ((int)hkv * KC);
          const int h = r / KC, c = r % KC;
          const long long src = s_src[i];
          if (src >= 0) {
            const long long slot = s_dst[i];
            const PairChunk pc = pair_chunk(c, HALF, style);
            const __nv_bfloat16 *s = kp + ((size_t)src * hkv + h) * D;
            va[u] = ld_stream(s + pc.off_a);
            vb[u] = ld_stream(s + pc.off_b);
            dst[u] = (((slot >> 4) * (long long)hkv + h) * 16 + (slot & 15)) * D;
            tab[u] = s_tab[i];
            chunk[u] = c;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (dst[u] < 0) continue;
        const int c = chunk[u];
        float2 cs[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) cs[q] = s_cs[tab[u]][8 * c + q];
        float x[8], y[8], uu[8], ww[8];
        unpack8(va[u], x);
        unpack8(vb[u], y);
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
        st_global16(kc + dst[u] + pc.off_a, pack8(x));
        st_global16(kc + dst[u] + pc.off_b, pack8(y));
      }
    }
  }
}

}  // namespace
}  // namespace pic

extern "C" pic_status_t pic_relocate(
    const pic_geom_t *geom, int32_t batch, int32_t max_docs, int32_t n_pool_docs,
    const void *k_pool, const void *v_pool, int64_t pool_tokens, const int64_t *doc_token_start,
    const int32_t *doc_len, const int32_t *req_doc_ids, const int32_t *req_num_docs,
    const int32_t *doc_offset, const int32_t *doc_delta, const int64_t *slot_mapping,
    int32_t max_ctx, int64_t num_pages, void *k_cache, void *v_cache, int32_t layer_begin,
    int32_t layer_end, pic_stream_t stream) {
  using namespace pic;
  RopeParams rp;
  pic_status_t st = make_rope(geom, &rp);
  if (st != PIC_OK) return st;
  if (max_docs == 0 && batch > 0) return PIC_OK;  // no document to move
  if (batch <= 0 || max_docs < 0 || n_pool_docs <= 0 || pool_tokens <= 0 || max_ctx <= 0 ||
      num_pages <= 0)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: sizes must be positive");
  if (layer_begin < 0 || layer_end > geom->num_layers || layer_begin >= layer_end)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: layer range [%d, %d) outside [0, %d)",
                layer_begin, layer_end, geom->num_layers);
  if (layer_end - layer_begin > 65535) return fail(PIC_ERR_INVALID_ARG, "pic_relocate: too many layers");
  if (!k_pool || !v_pool || !doc_token_start || !doc_len || !req_doc_ids || !req_num_docs ||
      !doc_offset || !doc_delta || !slot_mapping || !k_cache || !v_cache)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: NULL tensor");
  if ((reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
       reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_relocate: K/V tensors must be 16-byte aligned");
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_relocate: no device status word");

  RelocArgs a;
  a.max_docs = max_docs;
  a.n_pool = n_pool_docs;
  a.max_ctx = max_ctx;
  a.hkv = geom->num_kv_heads;
  a.layer_begin = layer_begin;
  a.pool_tokens = pool_tokens;
  a.num_pages = num_pages;
  a.k_pool = static_cast<const __nv_bfloat16 *>(k_pool);
  a.v_pool = static_cast<const __nv_bfloat16 *>(v_pool);
  a.doc_start = doc_token_start;
  a.doc_len = doc_len;
  a.ids = req_doc_ids;
  a.num_docs = req_num_docs;
  a.offset = doc_offset;
  a.slots = slot_mapping;
  a.delta = doc_delta;
  a.k_cache = static_cast<__nv_bfloat16 *>(k_cache);
  a.v_cache = static_cast<__nv_bfloat16 *>(v_cache);
  a.status = status;
  dim3 grid((max_ctx + kTok - 1) / kTok, batch, layer_end - layer_begin);
  if (grid.y > 65535) return fail(PIC_ERR_INVALID_ARG, "pic_relocate: batch too large");
  if (geom->head_dim == 128)
    relocate_kernel<128><<<grid, kThreads, 0, stream>>>(a, rp);
  else
    relocate_kernel<64><<<grid, kThreads, 0, stream>>>(a, rp);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_relocate launch");
  return PIC_OK;
}
