// pic_compose: the link operator's logical layout and slot map.
//
// SemPIC, "Background: Position-Independent Caching" (Eqs. 1-2): a request is
// P, D_1, S_1, ..., D_m, S_m, Q in canonical order (the post-document inline
// spans S_k may be empty) and the link operator R assigns each prepared
// document its final logical positions, interleaved with the spans; appendix
// "Logical Layout and Re-Rotation": at link time each logical prompt position
// is tied to the physical cache slot that holds it.
//
// One grid row per request.  Every CTA of a row re-derives the document
// offsets with block-wide prefix sums over the document and span lengths
// (loaded in parallel, kept in shared memory), then fills its 1024-position
// slice of the slot map and of the token map (source pool row and document
// index of every document position, found by binary search over the
// offsets).  Only the first CTA of a row writes the per-document outputs, the
// inline positions and ctx_len, and records device-side check failures.
#include "pic_internal.cuh"

namespace pic {
namespace {

constexpr int kThreads = 256;
constexpr int kPerThread = 4;
constexpr int kSlotsPerCta = kThreads * kPerThread;
constexpr int kMaxDocs = 8192;  // per request (shared-memory offsets)

struct ComposeArgs {
  int batch, max_docs, n_pool, max_pages, max_ctx, max_inline, page;
  long long num_pages;
  const int32_t *doc_len, *doc_base, *ids, *num_docs, *spans, *prefix, *query, *block_table;
  const int64_t *doc_start;
  int32_t *doc_offset, *doc_delta, *inline_pos, *ctx_len;
  int64_t *slot_mapping, *tok_map;
  int32_t *status;
};

// Inclusive block scan of one value per thread (kThreads threads).
__device__ long long block_inclusive_scan(long long v, long long *warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    long long t = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += t;
  }
  if (lane == 31) warp_tot[warp] = v;
  __syncthreads();
  long long add = 0;
  for (int w = 0; w < warp; ++w) add += warp_tot[w];
  __syncthreads();
  return v + add;
}

__global__ void __launch_bounds__(kThreads) compose_kernel(ComposeArgs a) {
  pdl_entry();
  const int b = blockIdx.y;
  const int tid = threadIdx.x;
  const bool lead = blockIdx.x == 0;
  __shared__ long long warp_tot[kThreads / 32];
  __shared__ long long s_carry;
  __shared__ int s_err, s_err_detail;
  extern __shared__ long long s_dyn[];
  long long *s_start = s_dyn;                                             // [max_docs]
  int32_t *s_off = reinterpret_cast<int32_t *>(s_dyn + a.max_docs);     // [max_docs]
  int32_t *s_len = s_off + a.max_docs;   // document lengths
  int32_t *s_sin = s_len + a.max_docs;   // inline index of each span's first token
  __shared__ long long s_scarry;
  if (tid == 0) {
    s_carry = 0;
    s_scarry = 0;
    s_err = 0;
    s_err_detail = b;
  }
  __syncthreads();

  const int P = a.prefix[b], Tq = a.query[b], m = a.num_docs[b];
  if (P < 0 || Tq < 0 || m < 0 || m > a.max_docs) {
    if (lead && tid == 0) {
      dev_fail(a.status, PIC_DEV_BAD_REQUEST, b);
      a.ctx_len[b] = -1;
    }
    return;
  }

  for (int k0 = 0; k0 < m; k0 += kThreads) {
    const int k = k0 + tid;
    long long n = 0, sp = 0, base = 0, start = 0;
    if (k < m) {
      const int id = a.ids[(size_t)b * a.max_docs + k];
      if (a.spans) {
        sp = a.spans[(size_t)b * a.max_docs + k];
        if (sp < 0) {
          atomicCAS(&s_err, 0, PIC_DEV_BAD_REQUEST);
          sp = 0;
        }
      }
      if (id < 0 || id >= a.n_pool) {
        atomicCAS(&s_err, 0, PIC_DEV_BAD_DOC_ID);
      } else {
        n = a.doc_len[id];
        base = a.doc_base[id];
        start = a.doc_start[id];
        if (n <= 0) {
          atomicCAS(&s_err, 0, PIC_DEV_BAD_DOC_LEN);
          n = 0;
        }
      }
    }
    // document k starts after the documents and spans before it
    const long long incl = block_inclusive_scan(n + sp, warp_tot);
    const long long off = P + s_carry + incl - (n + sp);
    const long long sincl = block_inclusive_scan(sp, warp_tot);
    if (k < m) {
      s_off[k] = (int32_t)off;
      s_start[k] = start;
      s_len[k] = (int32_t)n;
      s_sin[k] = (int32_t)(P + s_scarry + sincl - sp);
    }
    if (lead && k < m) {
      a.doc_offset[(size_t)b * a.max_docs + k] = (int32_t)off;
      a.doc_delta[(size_t)b * a.max_docs + k] = (int32_t)(off - base);
    }
    __syncthreads();
    if (tid == kThreads - 1) {
      s_carry += incl;
      s_scarry += sincl;
    }
    __syncthreads();
  }
  if (lead)
    for (int k = m + tid; k < a.max_docs; k += kThreads) {
      a.doc_offset[(size_t)b * a.max_docs + k] = -1;
      a.doc_delta[(size_t)b * a.max_docs + k] = 0;
    }

  const long long ctx = (long long)P + s_carry + Tq;
  const long long n_span = s_scarry;  // inline tokens in the spans
  if (tid == 0) {
    if (ctx > a.max_ctx || P + n_span + Tq > a.max_inline) atomicCAS(&s_err, 0, PIC_DEV_CTX_OVERFLOW);
    else if ((ctx + a.page - 1) / a.page > a.max_pages)
      atomicCAS(&s_err, 0, PIC_DEV_BLOCK_TABLE_SHORT);
  }
  __syncthreads();
  const int err = s_err;

  // Slot map and token map of this CTA's positions (beyond ctx: -1).
  const long long t_begin = (long long)blockIdx.x * kSlotsPerCta;
  int64_t *slots = a.slot_mapping + (size_t)b * a.max_ctx;
  int64_t *tmap = a.tok_map + (size_t)b * a.max_ctx;
  const int32_t *bt = a.block_table + (size_t)b * a.max_pages;
  const long long span_end = ctx - Tq;  // documents and spans occupy [P, span_end)
  int page[kPerThread];
#pragma unroll
  for (int u = 0; u < kPerThread; ++u) {  // independent loads first
    const long long t = t_begin + tid + u * kThreads;
    page[u] = (!err && t < ctx) ? bt[t / a.page] : -2;
  }
#pragma unroll
  for (int u = 0; u < kPerThread; ++u) {
    const long long t = t_begin + tid + u * kThreads;
    if (t >= a.max_ctx) continue;
    long long sl = -1, tm = -1;
    if (page[u] != -2) {
      if (page[u] < 0 || page[u] >= a.num_pages) atomicCAS(&s_err, 0, PIC_DEV_BAD_PAGE);
      else sl = (long long)page[u] * a.page + t % a.page;
      if (t >= P && t < span_end) {  // last doc whose offset <= t; its token unless in its span
        int lo = 0, hi = m - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (s_off[mid] <= t) lo = mid;
          else hi = mid - 1;
        }
        if (t < (long long)s_off[lo] + s_len[lo])
          tm = ((long long)lo << 40) | (s_start[lo] + (t - s_off[lo]));
      }
    }
    slots[t] = sl;
    tmap[t] = tm;
  }
  if (lead) {  // inline tokens in order: prefix, spans S_1..S_m, query
    int32_t *ip = a.inline_pos + (size_t)b * a.max_inline;
    for (int i = tid; i < a.max_inline; i += kThreads) {
      int v = -1;
      if (!err && i < P) {
        v = i;
      } else if (!err && i < P + n_span) {  // the last span starting at or before i holds it
        int lo = 0, hi = m - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (s_sin[mid] <= i) lo = mid;
          else hi = mid - 1;
        }
        v = s_off[lo] + s_len[lo] + (i - s_sin[lo]);
      } else if (!err && i < P + n_span + Tq) {
        v = (int)(ctx - Tq + (i - P - n_span));
      }
      ip[i] = v;
    }
  }
  __syncthreads();
  if (tid == 0 && s_err) dev_fail(a.status, s_err, s_err_detail);
  if (lead && tid == 0) a.ctx_len[b] = s_err ? -1 : (int32_t)ctx;
}

}  // namespace
}  // namespace pic

extern "C" pic_status_t pic_compose(const pic_geom_t *geom, int32_t batch, int32_t max_docs,
                                    int32_t n_pool_docs, const int32_t *doc_len,
                                    const int32_t *doc_base_pos, const int64_t *doc_token_start,
                                    const int32_t *req_doc_ids,
                                    const int32_t *req_num_docs, const int32_t *span_len,
                                    const int32_t *prefix_len,
                                    const int32_t *query_len, const int32_t *block_table,
                                    int32_t max_pages, int64_t num_pages, int32_t max_ctx,
                                    int32_t max_inline, int32_t *doc_offset, int32_t *doc_delta,
                                    int64_t *slot_mapping, int64_t *tok_map,
                                    int32_t *inline_pos, int32_t *ctx_len, pic_stream_t stream) {
  using namespace pic;
  double theta[kMaxHalfDim];
  pic_status_t st = check_geom(geom, theta);
  if (st != PIC_OK) return st;
  if (batch <= 0 || max_docs < 0 || n_pool_docs < 0 || max_pages <= 0 || num_pages <= 0 ||
      max_ctx <= 0 || max_inline <= 0)
    return fail(PIC_ERR_INVALID_ARG, "pic_compose: sizes must be positive");
  if (num_pages > (int64_t)INT32_MAX)
    return fail(PIC_ERR_INVALID_ARG, "pic_compose: num_pages exceeds int32");
  if (!doc_len || !doc_base_pos || !doc_token_start || !req_num_docs || !prefix_len ||
      !query_len || !block_table || !slot_mapping || !tok_map || !inline_pos || !ctx_len ||
      (max_docs > 0 && (!req_doc_ids || !doc_offset || !doc_delta)))
    return fail(PIC_ERR_INVALID_ARG, "pic_compose: NULL tensor");
  if (max_docs > kMaxDocs)
    return fail(PIC_ERR_UNSUPPORTED, "pic_compose: max_docs %d > %d", max_docs, kMaxDocs);
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_compose: no device status word");
  ComposeArgs a;
  a.batch = batch;
  a.max_docs = max_docs;
  a.n_pool = n_pool_docs;
  a.max_pages = max_pages;
  a.max_ctx = max_ctx;
  a.max_inline = max_inline;
  a.page = geom->page_size;
  a.num_pages = num_pages;
  a.doc_len = doc_len;
  a.doc_base = doc_base_pos;
  a.doc_start = doc_token_start;
  a.ids = req_doc_ids;
  a.num_docs = req_num_docs;
  a.spans = max_docs > 0 ? span_len : nullptr;
  a.prefix = prefix_len;
  a.query = query_len;
  a.block_table = block_table;
  a.doc_offset = doc_offset;
  a.doc_delta = doc_delta;
  a.inline_pos = inline_pos;
  a.ctx_len = ctx_len;
  a.slot_mapping = slot_mapping;
  a.tok_map = tok_map;
  a.status = status;
  dim3 grid((max_ctx + kSlotsPerCta - 1) / kSlotsPerCta, batch);
  const size_t smem = (size_t)max_docs * (sizeof(long long) + 3 * sizeof(int32_t)) + 16;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(compose_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return cuda_fail(e, "pic_compose smem attribute");
  }
  cudaError_t le = launch_dependent(compose_kernel, grid, dim3(kThreads), smem, stream, a);
  if (le != cudaSuccess) return cuda_fail(le, "pic_compose launch");
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_compose launch");
  return PIC_OK;
}
