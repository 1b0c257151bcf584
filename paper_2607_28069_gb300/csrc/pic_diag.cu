// pic_attention_deviation: the attention-deviation diagnostic of SemPIC's
// "Motivating Analysis" -- the mean absolute deviation between the
// post-softmax attention probabilities of two configurations A and B within
// normalized block regions (pre = [0, 0.1), int = [0.1, 0.9) of each reusable
// block).  Here A and B are two stitched key caches of the same requests
// with the same slot map (e.g. relocated documents, and documents left at
// their compiled positions), read by the same rotated queries.
//
// One CTA per (128-key chunk of the logical positions, kv head, request).
// It gathers the chunk's K rows of both caches through the slot map into
// shared memory, keeps the region of every document key (the normalized
// position of token j of a block of n tokens is j / n; region i holds
// ceil(e_i n) <= j < ceil(e_(i+1) n)), then streams the request's query
// rows of that kv head (the last query_len inline tokens, every query head
// of the group, 64 rows at a time from the packed-query workspace):
// p_X = exp(q.k_X / sqrt(d) - lse_X) with lse_X the log-sum-exp of the
// prefill attention of configuration X, and |p_A - p_B| summed per region.
// A diagnostic off the serving path: CUDA-core FMAs, fp32 terms, fp64 sums.
#include "pic_internal.cuh"

namespace pic {
namespace {

constexpr int kThreads = 256;
constexpr int kKeys = 128;   // key positions per CTA
constexpr int kRows = 64;    // query rows per pass
constexpr int kMaxRegions = 8;

struct DevArgs {
  int Hq, Hkv, G, max_inline, max_docs, max_ctx, R_pad, n_regions;
  long long num_pages, layer_row0;
  const int32_t *inline_pos, *inline_len, *query_len, *ids, *doc_len, *doc_offset;
  const int64_t *slots, *tok_map;
  const __nv_bfloat16 *ka, *kb, *qpack;
  const float *lse_a, *lse_b;
  double edges[kMaxRegions + 1];
  double *sums;
  unsigned long long *counts;
  float scale;
};

template <int D>
__global__ void __launch_bounds__(kThreads) deviation_kernel(DevArgs a) {
  constexpr int C8 = D / 8;  // 16-byte chunks per row
  const int b = blockIdx.z, hk = blockIdx.y, tid = threadIdx.x;
  const long long t0 = (long long)blockIdx.x * kKeys;
  // K rows of both caches and the query rows: 80 KB at d = 128 (dynamic)
  extern __shared__ __align__(16) uint8_t s_dyn[];
  auto s_ka = reinterpret_cast<__nv_bfloat16 (*)[D]>(s_dyn);
  auto s_kb = reinterpret_cast<__nv_bfloat16 (*)[D]>(s_dyn + kKeys * D * 2);
  auto s_q = reinterpret_cast<__nv_bfloat16 (*)[D]>(s_dyn + 2 * kKeys * D * 2);
  __shared__ int s_reg[kKeys];     // region of the key (-1: not a block token of a region)
  __shared__ int s_pos[kKeys];     // logical position
  __shared__ float s_la[kRows], s_lb[kRows];
  __shared__ int s_rpos[kRows];
  __shared__ double s_sum[kMaxRegions];
  __shared__ unsigned long long s_cnt[kMaxRegions];
  __shared__ int s_any;

  const int tin = min(max(a.inline_len[b], 0), a.max_inline);
  const int tq = min(max(a.query_len[b], 0), tin);
  if (tid < kMaxRegions) {
    s_sum[tid] = 0.0;
    s_cnt[tid] = 0ull;
  }
  if (tid == 0) s_any = 0;
  __syncthreads();

  // ---- the chunk's keys: region and the K rows of both caches
  if (tid < kKeys) {
    const long long t = t0 + tid;
    int reg = -1;
    if (t < a.max_ctx) {
      const long long tm = a.tok_map[(size_t)b * a.max_ctx + t];
      if (tm >= 0) {
        const int k = (int)(tm >> 40);
        const int id = k < a.max_docs ? a.ids[(size_t)b * a.max_docs + k] : -1;
        const int n = id >= 0 ? a.doc_len[id] : 0;
        const long long j = t - a.doc_offset[(size_t)b * a.max_docs + (k < a.max_docs ? k : 0)];
        for (int i = 0; i < a.n_regions && n > 0; ++i)
          if (j >= (long long)ceil(a.edges[i] * n) && j < (long long)ceil(a.edges[i + 1] * n)) reg = i;
      }
    }
    s_reg[tid] = reg;
    s_pos[tid] = (int)t;
    if (reg >= 0) {
      atomicAdd(&s_cnt[reg], (unsigned long long)tq * a.G);
      s_any = 1;
    }
  }
  __syncthreads();
  if (!s_any || tq == 0) {  // nothing of a region here
    if (tid < a.n_regions && s_cnt[tid])
      atomicAdd(&a.counts[(size_t)b * a.n_regions + tid], s_cnt[tid]);
    return;
  }
  for (int e = tid; e < kKeys * C8; e += kThreads) {
    const int key = e / C8, c = e % C8;
    uint4 va = make_uint4(0, 0, 0, 0), vb = va;
    if (s_reg[key] >= 0) {
      const long long slot = a.slots[(size_t)b * a.max_ctx + t0 + key];
      if (slot >= 0 && (slot >> 4) < a.num_pages) {
        const size_t row = (size_t)(a.layer_row0 + ((slot >> 4) * a.Hkv + hk) * 16 + (slot & 15));
        va = *reinterpret_cast<const uint4 *>(a.ka + row * D + c * 8);
        vb = *reinterpret_cast<const uint4 *>(a.kb + row * D + c * 8);
      }
    }
    *reinterpret_cast<uint4 *>(&s_ka[key][c * 8]) = va;
    *reinterpret_cast<uint4 *>(&s_kb[key][c * 8]) = vb;
  }

  // ---- query rows of this kv head: inline tokens tin - tq .. tin - 1, all G heads
  const int row_begin = (tin - tq) * a.G, row_end = tin * a.G;
  const int my_row = tid >> 2;  // 4 threads per row, keys tid & 3, + 4, + 8, ...
  float part[kMaxRegions];
#pragma unroll
  for (int i = 0; i < kMaxRegions; ++i) part[i] = 0.f;
  for (int r0 = row_begin; r0 < row_end; r0 += kRows) {
    __syncthreads();  // previous rows consumed (and the K rows above written)
    for (int e = tid; e < kRows * C8; e += kThreads) {
      const int r = e / C8, c = e % C8;
      uint4 v = make_uint4(0, 0, 0, 0);
      if (r0 + r < row_end)
        v = *reinterpret_cast<const uint4 *>(
            a.qpack + (((size_t)b * a.Hkv + hk) * a.R_pad + r0 + r) * D + c * 8);
      *reinterpret_cast<uint4 *>(&s_q[r][c * 8]) = v;
    }
    if (tid < kRows) {
      const int rg = r0 + tid;
      float la = 0.f, lb = 0.f;
      int pos = -1;
      if (rg < row_end) {
        const int tok = rg / a.G, h = hk * a.G + rg % a.G;
        const size_t li = ((size_t)b * a.max_inline + tok) * a.Hq + h;
        la = a.lse_a[li];
        lb = a.lse_b[li];
        pos = a.inline_pos[(size_t)b * a.max_inline + tok];
      }
      s_la[tid] = la;
      s_lb[tid] = lb;
      s_rpos[tid] = pos;
    }
    __syncthreads();
    if (r0 + my_row >= row_end) continue;
    float acc_a[kKeys / 4], acc_b[kKeys / 4];
#pragma unroll
    for (int m = 0; m < kKeys / 4; ++m) acc_a[m] = acc_b[m] = 0.f;
#pragma unroll 1
    for (int c = 0; c < C8; ++c) {
      float qv[8];
      unpack8(*reinterpret_cast<const uint4 *>(&s_q[my_row][c * 8]), qv);
#pragma unroll
      for (int m = 0; m < kKeys / 4; ++m) {
        const int key = (tid & 3) + 4 * m;
        float x[8], y[8];
        unpack8(*reinterpret_cast<const uint4 *>(&s_ka[key][c * 8]), x);
        unpack8(*reinterpret_cast<const uint4 *>(&s_kb[key][c * 8]), y);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          acc_a[m] = fmaf(qv[i], x[i], acc_a[m]);
          acc_b[m] = fmaf(qv[i], y[i], acc_b[m]);
        }
      }
    }
    const float la = s_la[my_row], lb = s_lb[my_row];
    const int rpos = s_rpos[my_row];
#pragma unroll
    for (int m = 0; m < kKeys / 4; ++m) {
      const int key = (tid & 3) + 4 * m;
      const int reg = s_reg[key];
      if (reg < 0 || s_pos[key] > rpos) continue;  // not in a region, or not visible
      const float pa = expf(acc_a[m] * a.scale - la), pb = expf(acc_b[m] * a.scale - lb);
      const float dv = fabsf(pa - pb);
#pragma unroll
      for (int i = 0; i < kMaxRegions; ++i)
        if (i == reg) part[i] += dv;
    }
  }
  // ---- reduce: warp, then shared, then one global add per region
#pragma unroll
  for (int i = 0; i < kMaxRegions; ++i) {
    double v = part[i];
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((tid & 31) == 0 && v != 0.0) atomicAdd(&s_sum[i], v);
  }
  __syncthreads();
  if (tid < a.n_regions) {
    if (s_sum[tid] != 0.0) atomicAdd(&a.sums[(size_t)b * a.n_regions + tid], s_sum[tid]);
    if (s_cnt[tid]) atomicAdd(&a.counts[(size_t)b * a.n_regions + tid], s_cnt[tid]);
  }
}

}  // namespace
}  // namespace pic

extern "C" pic_status_t pic_attention_deviation(
    const pic_geom_t *geom, int32_t layer, int32_t batch, int32_t max_inline, int32_t max_docs,
    int32_t max_ctx, int64_t num_pages, const int32_t *inline_pos, const int32_t *inline_len,
    const int32_t *query_len, const int32_t *req_doc_ids, const int32_t *doc_len,
    const int32_t *doc_offset, const int64_t *slot_mapping, const int64_t *tok_map,
    const void *k_cache_a, const void *k_cache_b, const float *lse_a, const float *lse_b,
    const double *edges, int32_t n_regions, const void *workspace, size_t workspace_bytes,
    double *sums, int64_t *counts, pic_stream_t stream) {
  using namespace pic;
  double theta[kMaxHalfDim];
  pic_status_t st = check_geom(geom, theta);
  if (st != PIC_OK) return st;
  if (layer < 0 || layer >= geom->num_layers)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: layer %d outside [0, %d)", layer,
                geom->num_layers);
  if (batch <= 0 || max_inline <= 0 || max_docs <= 0 || max_ctx <= 0 || num_pages <= 0)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: sizes must be positive");
  if (n_regions < 1 || n_regions > kMaxRegions || !edges)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: 1..%d regions", kMaxRegions);
  for (int i = 0; i <= n_regions; ++i) {
    if (!(edges[i] >= 0.0 && edges[i] <= 1.0) || (i > 0 && !(edges[i] >= edges[i - 1])))
      return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: edges must ascend in [0, 1]");
  }
  if (!inline_pos || !inline_len || !query_len || !req_doc_ids || !doc_len || !doc_offset ||
      !slot_mapping || !tok_map || !k_cache_a || !k_cache_b || !lse_a || !lse_b || !workspace ||
      !sums || !counts)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: NULL tensor");
  const int Hkv = geom->num_kv_heads, G = geom->num_q_heads / Hkv, D = geom->head_dim;
  const long long m_tiles = ((long long)max_inline * G + 127) / 128;
  const long long R_pad = m_tiles * 128;
  if ((size_t)batch * Hkv * R_pad * D * 2 > workspace_bytes)
    return fail(PIC_ERR_WORKSPACE, "pic_attention_deviation: workspace smaller than the packed queries");
  if ((reinterpret_cast<uintptr_t>(k_cache_a) | reinterpret_cast<uintptr_t>(k_cache_b) |
       reinterpret_cast<uintptr_t>(workspace)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: bf16 tensors must be 16-byte aligned");
  if (batch > 65535 || Hkv > 65535)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: grid too large");
  DevArgs a;
  a.Hq = geom->num_q_heads;
  a.Hkv = Hkv;
  a.G = G;
  a.max_inline = max_inline;
  a.max_docs = max_docs;
  a.max_ctx = max_ctx;
  a.R_pad = (int)R_pad;
  a.n_regions = n_regions;
  a.num_pages = num_pages;
  a.layer_row0 = (long long)layer * num_pages * Hkv * 16;
  a.inline_pos = inline_pos;
  a.inline_len = inline_len;
  a.query_len = query_len;
  a.ids = req_doc_ids;
  a.doc_len = doc_len;
  a.doc_offset = doc_offset;
  a.slots = slot_mapping;
  a.tok_map = tok_map;
  a.ka = static_cast<const __nv_bfloat16 *>(k_cache_a);
  a.kb = static_cast<const __nv_bfloat16 *>(k_cache_b);
  a.qpack = static_cast<const __nv_bfloat16 *>(workspace);
  a.lse_a = lse_a;
  a.lse_b = lse_b;
  for (int i = 0; i <= kMaxRegions; ++i) a.edges[i] = i <= n_regions ? edges[i] : 1.0;
  a.sums = sums;
  a.counts = reinterpret_cast<unsigned long long *>(counts);
  a.scale = (float)(1.0 / std::sqrt((double)D));
  cudaError_t e = cudaMemsetAsync(sums, 0, sizeof(double) * batch * n_regions, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(counts, 0, sizeof(int64_t) * batch * n_regions, stream);
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation clear");
  const dim3 grid((unsigned)((max_ctx + kKeys - 1) / kKeys), Hkv, batch);
  const int smem = (2 * kKeys + kRows) * D * 2;
  if (D == 128) {
    e = cudaFuncSetAttribute(deviation_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) deviation_kernel<128><<<grid, kThreads, smem, stream>>>(a);
  } else {
    e = cudaFuncSetAttribute(deviation_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) deviation_kernel<64><<<grid, kThreads, smem, stream>>>(a);
  }
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation smem attribute");
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation launch");
  return PIC_OK;
}
