// pic_attention_deviation: the attention-deviation diagnostic of SemPIC's
// "Motivating Analysis" -- the mean absolute deviation between the
// post-softmax attention probabilities of two configurations A and B within
// normalized block regions (pre = [0, 0.1), int = [0.1, 0.9) of each reusable
// block).  Here A and B are two stitched key caches of the same requests
// with the same slot map (e.g. relocated documents, and documents left at
// their compiled positions), read by the same rotated queries.
//
// Both score matrices are dense contractions (S_X = Q K_X^T over the
// documents' keys), so they run on the tensor cores (tcgen05, scores in
// TMEM); the normalized position of token j of a block of n tokens is j / n
// and region i holds ceil(e_i n) <= j < ceil(e_(i+1) n).  The query rows
// are the request's last query_len inline tokens, every query head of the
// group, from the packed-query workspace; p_X = exp(q.k_X / sqrt(d) - lse_X)
// with lse_X the log-sum-exp of the prefill attention of configuration X,
// and |p_A - p_B| is summed per region (fp32 terms, fp64 sums).
#include "pic_internal.cuh"

namespace pic {
namespace {

constexpr int kThreads = 320;  // warp 0 TMA producer, warp 1 MMA issuer, warps 2-9 compute
constexpr int kComputeWarps = 8;  // two per TMEM lane quarter, each on half the key columns
constexpr int BM = 128;        // query rows per tile (TMEM lanes)
constexpr int BN = 128;        // key positions per tile
constexpr int NS = 2;          // K stages, each a tile of cache A and one of cache B
constexpr int kMaxRegions = 8;
constexpr uint32_t kTmemCols = 512;  // two buffers of (S_A, S_B), 128 columns each

template <int D>
struct DLayout {
  static constexpr int kTile = BN * D * 2;        // one K tile
  static constexpr int kQ = 0;
  static constexpr int kK = kQ + BM * D * 2;      // stage st: A at kK + 2 st kTile, B after it
  static constexpr int kReg = kK + NS * 2 * kTile;  // int8 region of each key, [2][BN]
  static constexpr int kBar = kReg + 2 * BN;
  static constexpr int kBytes = kBar + 256;
  static constexpr int kAlloc = kBytes + 1024;
};

enum {
  DB_Q = 0,
  DB_KFULL = 1,
  DB_KEMPTY = DB_KFULL + NS,
  DB_SFULL = DB_KEMPTY + NS,  // per S buffer
  DB_SFREE = DB_SFULL + 2,    // per S buffer, one arrival per compute warp
  DB_FINAL = DB_SFREE + 2,
  DB_COUNT = DB_FINAL + 1
};

struct DevArgs {
  int Hq, Hkv, G, max_inline, max_docs, max_ctx, R_pad, n_regions, splits;
  long long num_pages, layer_row0, oob_row;
  const int32_t *inline_pos, *inline_len, *query_len, *ids, *doc_len, *doc_offset;
  const int64_t *slots, *tok_map;
  const float *lse_a, *lse_b;
  double edges[kMaxRegions + 1];
  double *sums;
  unsigned long long *counts;
  int32_t *status;
  float scale_log2;
};

// Region of the document token at logical position t of request b (-1: not
// a document token, or in no region).
__device__ int key_region(const DevArgs &a, int b, long long t) {
  if (t < 0 || t >= a.max_ctx) return -1;
  const long long tm = a.tok_map[(size_t)b * a.max_ctx + t];
  if (tm < 0) return -1;
  const int k = (int)(tm >> 40);
  if (k >= a.max_docs) return -1;
  const int id = a.ids[(size_t)b * a.max_docs + k];
  const int n = id >= 0 ? a.doc_len[id] : 0;
  const long long j = t - a.doc_offset[(size_t)b * a.max_docs + k];
  int reg = -1;
  for (int i = 0; i < a.n_regions && n > 0; ++i)
    if (j >= (long long)ceil(a.edges[i] * n) && j < (long long)ceil(a.edges[i + 1] * n)) reg = i;
  return reg;
}

// CTA = (128-row query tile, key split, kv head, request).  Per 128-key tile
// of the documents' span: the producer loads the tile of both caches (page
// boxes through the block layout, as the prefill attention does) and writes
// the key regions; the issuer computes S_A = Q K_A^T and S_B = Q K_B^T into a
// TMEM buffer (two buffers, so the next tile's MMAs overlap this one's
// exponentials); each compute thread owns one query row, reads both rows of
// scores from TMEM 32 columns at a time and adds |p_A - p_B| to its region.
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    deviation_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_ka,
                     const __grid_constant__ CUtensorMap tm_kb, DevArgs a) {
  using L = DLayout<D>;
  constexpr int PANELS = D / 64;
  constexpr uint32_t IDESC_QK = idesc_bf16(BM, BN, false, false);
  constexpr uint32_t kPageBytes = 16 * D * 2;
  constexpr uint32_t kGroupStride = PANELS == 2 ? 2048 : 1024;
  constexpr uint32_t kPanelOff = PANELS == 2 ? 1024 : BN * 128;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  auto bar = [&](int i) { return sbase + L::kBar + 8u * (uint32_t)i; };
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + L::kBar + 8 * DB_COUNT);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::kBar + 8 * DB_COUNT + 8);
  int8_t *s_reg = reinterpret_cast<int8_t *>(smem + L::kReg);
  __shared__ double s_sum[kMaxRegions];
  __shared__ int s_m;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int qt = blockIdx.x / a.splits, split = blockIdx.x % a.splits;
  const int hk = blockIdx.y, b = blockIdx.z;

  if (tid == 0) {
    for (int i = 0; i < DB_COUNT; ++i)
      mbar_init(bar(i), (i == DB_SFREE || i == DB_SFREE + 1) ? kComputeWarps : 1);
    *abort_flag = 0;
    fence_mbar_init();
    int m = 0;  // documents of the request: doc_offset is -1 past them
    while (m < a.max_docs && a.doc_offset[(size_t)b * a.max_docs + m] >= 0) ++m;
    s_m = m;
  }
  if (tid < kMaxRegions) s_sum[tid] = 0.0;
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tmem_slot;

  // ---- the work of this CTA (uniform)
  const int tin = min(max(a.inline_len[b], 0), a.max_inline);
  const int tq = min(max(a.query_len[b], 0), tin);
  const int row_begin = (tin - tq) * a.G, row_end = tin * a.G;
  const int r0 = row_begin + qt * BM;
  const int m = s_m;
  long long key_lo = 0, key_hi = 0;
  if (m > 0) {
    key_lo = a.doc_offset[(size_t)b * a.max_docs];
    const int id = a.ids[(size_t)b * a.max_docs + m - 1];
    key_hi = a.doc_offset[(size_t)b * a.max_docs + m - 1] + (id >= 0 ? a.doc_len[id] : 0);
  }
  const int kt0 = (int)(key_lo / BN);
  const int n_kt = key_hi > key_lo ? (int)((key_hi - 1) / BN) - kt0 + 1 : 0;
  const int per = (n_kt + a.splits - 1) / a.splits;
  const int kv_begin = split * per;
  const int n = max(0, min(per, n_kt - kv_begin));

  // the number of terms of each region: one CTA per request
  if (qt == 0 && split == 0 && hk == 0 && warp >= 2)
    for (int k = tid - 64; k < m; k += 32 * kComputeWarps) {
      const int id = a.ids[(size_t)b * a.max_docs + k];
      const int nk = id >= 0 ? a.doc_len[id] : 0;
      for (int i = 0; i < a.n_regions && nk > 0; ++i) {
        const long long lo = (long long)ceil(a.edges[i] * nk), hi = (long long)ceil(a.edges[i + 1] * nk);
        if (hi > lo)
          atomicAdd(&a.counts[(size_t)b * a.n_regions + i], (unsigned long long)(hi - lo) * tq * a.Hq);
      }
    }

  if (r0 < row_end && n > 0) {
    if (warp == 0) {
      // ================================================ TMA producer
      if (lane == 0) {
        prefetch_tmap(&tm_q);
        prefetch_tmap(&tm_ka);
        prefetch_tmap(&tm_kb);
        mbar_expect_tx(bar(DB_Q), BM * D * 2);
        const int qrow = (b * a.Hkv + hk) * a.R_pad + r0;
#pragma unroll
        for (int pn = 0; pn < PANELS; ++pn)
          tma_load_2d(sbase + L::kQ + pn * BM * 128, &tm_q, pn * 64, qrow, bar(DB_Q));
      }
      for (int j = 0; j < n; ++j) {
        const int st = j % NS, kt = kt0 + kv_begin + j;
        bool ok = true;
        if (j >= NS) ok = mbar_wait(bar(DB_KEMPTY + st), ((j / NS) - 1) & 1, abort_flag, a.status, b);
        if (ok && j >= 2) ok = mbar_wait(bar(DB_SFREE + (j & 1)), ((j >> 1) - 1) & 1, abort_flag, a.status, b);
        if (!__all_sync(0xffffffffu, ok)) break;
        for (int c = lane; c < BN; c += 32)
          s_reg[(j & 1) * BN + c] = (int8_t)key_region(a, b, (long long)kt * BN + c);
        int y = (int)a.oob_row;  // lanes 0..7: page row of page `lane` of the tile
        if (lane < 8) {
          const long long t = ((long long)kt * 8 + lane) * 16;
          const long long slot = t < a.max_ctx ? a.slots[(size_t)b * a.max_ctx + t] : -1;
          if (slot >= 0 && (slot >> 4) < a.num_pages)
            y = (int)(a.layer_row0 + ((slot >> 4) * a.Hkv + hk) * 16);
        }
        __syncwarp();
        if (lane == 0) mbar_expect_tx(bar(DB_KFULL + st), 2 * L::kTile);
        __syncwarp();
        if (lane < 8) {
          const uint32_t dst = sbase + L::kK + st * 2 * L::kTile + lane * kPageBytes;
          if constexpr (PANELS == 2) {
            tma_load_4d(dst, &tm_ka, 0, 0, 0, y >> 3, bar(DB_KFULL + st));
            tma_load_4d(dst + L::kTile, &tm_kb, 0, 0, 0, y >> 3, bar(DB_KFULL + st));
          } else {
            tma_load_2d(dst, &tm_ka, 0, y, bar(DB_KFULL + st));
            tma_load_2d(dst + L::kTile, &tm_kb, 0, y, bar(DB_KFULL + st));
          }
        }
      }
    } else if (warp == 1) {
      // ================================================ MMA issuer
      if (lane == 0) {
        bool ok = mbar_wait(bar(DB_Q), 0, abort_flag, a.status, b);
        tc_fence_after();
        const uint64_t dQ = sdesc_sw128(sbase + L::kQ, 16, 1024);
        const uint64_t dK = sdesc_sw128(sbase + L::kK, 16, kGroupStride);
        for (int j = 0; ok && j < n; ++j) {
          const int st = j % NS, buf = j & 1;
          ok = mbar_wait(bar(DB_KFULL + st), (j / NS) & 1, abort_flag, a.status, b);
          if (ok && j >= 2) ok = mbar_wait(bar(DB_SFREE + buf), ((j >> 1) - 1) & 1, abort_flag, a.status, b);
          if (!ok) break;
          tc_fence_after();
          const uint32_t tSA = tbase + buf * 256, tSB = tSA + 128;
          const uint64_t dka = dK + (uint64_t)((st * 2 * L::kTile) >> 4);
          const uint64_t dkb = dka + (uint64_t)(L::kTile >> 4);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t qd = dQ + ((kk >> 2) * (BM * 128) + (kk & 3) * 32) / 16;
            const uint64_t ko = ((kk >> 2) * kPanelOff + (kk & 3) * 32) / 16;
            mma_ss(tSA, qd, dka + ko, IDESC_QK, kk > 0);
            mma_ss(tSB, qd, dkb + ko, IDESC_QK, kk > 0);
          }
          mma_commit(bar(DB_SFULL + buf));
          mma_commit(bar(DB_KEMPTY + st));
        }
        mma_commit(bar(DB_FINAL));
      }
    } else {
      // ================================================ compute warps
      // Two warps per TMEM lane quarter, each on 64 of the 128 key columns.
      // Keys come in runs of one region (the producer's bytes, the same for
      // every row): |p_A - p_B| is summed per run and added to the run's
      // region when the region changes.  A key after a row's position (an
      // inline span taken as a query row before a later document) has
      // p_A = p_B = 0; 32-key chunks that every row of the warp sees skip
      // that test.
      const int wq = warp & 3, half = (warp - 2) >> 2;
      const int row = wq * 32 + lane, rg = r0 + row;
      float la = INFINITY, lb = INFINITY;  // rows past the query rows add nothing
      long long qpos = LLONG_MAX;
      if (rg < row_end) {
        const int tok = rg / a.G, h = hk * a.G + rg % a.G;
        const size_t li = ((size_t)b * a.max_inline + tok) * a.Hq + h;
        la = a.lse_a[li] * 1.4426950408889634f;
        lb = a.lse_b[li] * 1.4426950408889634f;
        qpos = a.inline_pos[(size_t)b * a.max_inline + tok];
      }
      long long wmin = qpos;
#pragma unroll
      for (int o = 16; o; o >>= 1) wmin = min(wmin, __shfl_xor_sync(0xffffffffu, wmin, o));
      const uint32_t tl = tbase + ((uint32_t)(wq * 32) << 16) + half * 64;
      float acc[kMaxRegions];
#pragma unroll
      for (int i = 0; i < kMaxRegions; ++i) acc[i] = 0.f;
      int cur = -1;
      float run = 0.f;
      auto flush = [&]() {
#pragma unroll
        for (int i = 0; i < kMaxRegions; ++i)
          if (i == cur) acc[i] += run;
        run = 0.f;
      };
      for (int j = 0; j < n; ++j) {
        const int st = j % NS, buf = j & 1;
        // K(j) landed (also publishes the producer's region bytes), S(j) ready
        bool ok = mbar_wait(bar(DB_KFULL + st), (j / NS) & 1, abort_flag, a.status, b);
        if (ok) ok = mbar_wait(bar(DB_SFULL + buf), (j >> 1) & 1, abort_flag, a.status, b);
        if (!__all_sync(0xffffffffu, ok)) break;
        tc_fence_after();
#pragma unroll 1
        for (int c0 = 0; c0 < 64; c0 += 32) {
          float sa[32], sb[32];
          tmem_ld32(tl + buf * 256 + c0, reinterpret_cast<uint32_t *>(sa));
          tmem_ld32(tl + buf * 256 + 128 + c0, reinterpret_cast<uint32_t *>(sb));
          tmem_wait_ld();
          const int8_t *rr = s_reg + buf * BN + half * 64 + c0;
          const long long t0 = (long long)(kt0 + kv_begin + j) * BN + half * 64 + c0;
          if (t0 + 31 <= wmin) {
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const int reg = rr[c];
              if (reg != cur) {  // the same for every thread: no divergence
                flush();
                cur = reg;
              }
              if (reg >= 0)
                run += fabsf(ex2(fmaf(sa[c], a.scale_log2, -la)) - ex2(fmaf(sb[c], a.scale_log2, -lb)));
            }
          } else {
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const int reg = rr[c];
              if (reg != cur) {
                flush();
                cur = reg;
              }
              if (reg >= 0 && t0 + c <= qpos)
                run += fabsf(ex2(fmaf(sa[c], a.scale_log2, -la)) - ex2(fmaf(sb[c], a.scale_log2, -lb)));
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(DB_SFREE + buf));
      }
      flush();
#pragma unroll
      for (int i = 0; i < kMaxRegions; ++i) {
        double v = acc[i];
#pragma unroll
        for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0 && v != 0.0) atomicAdd(&s_sum[i], v);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid < a.n_regions && s_sum[tid] != 0.0) atomicAdd(&a.sums[(size_t)b * a.n_regions + tid], s_sum[tid]);
  if (warp == 1) {
    tc_fence_after();
    if (r0 < row_end && n > 0 && lane == 0) mbar_wait(bar(DB_FINAL), 0, abort_flag, a.status, b);
    __syncwarp();
    tmem_dealloc(tbase, kTmemCols);
  }
}

}  // namespace
}  // namespace pic

extern "C" pic_status_t pic_attention_deviation(
    const pic_geom_t *geom, int32_t layer, int32_t batch, int32_t max_inline, int32_t max_docs,
    int32_t max_ctx, int64_t num_pages, const int32_t *inline_pos, const int32_t *inline_len,
    const int32_t *query_len, int32_t max_query_len, const int32_t *req_doc_ids,
    const int32_t *doc_len,
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
  if (max_query_len < 0 || max_query_len > max_inline)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: max_query_len outside [0, max_inline]");
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
  const long long rows_total = (long long)geom->num_layers * num_pages * Hkv * 16;
  if (rows_total + 16 >= (long long)INT32_MAX)
    return fail(PIC_ERR_UNSUPPORTED, "pic_attention_deviation: cache has more than 2^31 rows");
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_attention_deviation: no device status word");
  CUtensorMap tq, tka, tkb;
  st = encode_tmap_2d(&tq, workspace, D, (uint64_t)batch * Hkv * R_pad, (uint64_t)D * 2, 64, BM);
  if (D == 128) {
    if (st == PIC_OK) st = encode_tmap_pages128(&tka, k_cache_a, (uint64_t)rows_total / 16);
    if (st == PIC_OK) st = encode_tmap_pages128(&tkb, k_cache_b, (uint64_t)rows_total / 16);
  } else {
    if (st == PIC_OK) st = encode_tmap_2d(&tka, k_cache_a, D, rows_total, (uint64_t)D * 2, 64, 16);
    if (st == PIC_OK) st = encode_tmap_2d(&tkb, k_cache_b, D, rows_total, (uint64_t)D * 2, 64, 16);
  }
  if (st != PIC_OK) return st;
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
  a.oob_row = rows_total;
  a.inline_pos = inline_pos;
  a.inline_len = inline_len;
  a.query_len = query_len;
  a.ids = req_doc_ids;
  a.doc_len = doc_len;
  a.doc_offset = doc_offset;
  a.slots = slot_mapping;
  a.tok_map = tok_map;
  a.lse_a = lse_a;
  a.lse_b = lse_b;
  for (int i = 0; i <= kMaxRegions; ++i) a.edges[i] = i <= n_regions ? edges[i] : 1.0;
  a.sums = sums;
  a.counts = reinterpret_cast<unsigned long long *>(counts);
  a.status = status;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D));
  // query tiles: the query rows of a request are its last query_len inline
  // tokens times G; key splits: enough CTAs for two waves of the GPU (every
  // split adds its own partial sums)
  const int q_tiles = (int)(((long long)max_query_len * G + BM - 1) / BM);
  const int kt_max = (max_ctx + BN - 1) / BN;
  const long long groups = (long long)batch * Hkv * std::max(q_tiles, 1);
  a.splits = (int)std::max<long long>(1, std::min<long long>(std::min(kt_max, 64),
                                                             (2 * 152 + groups - 1) / groups));
  cudaError_t e = cudaMemsetAsync(sums, 0, sizeof(double) * batch * n_regions, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(counts, 0, sizeof(int64_t) * batch * n_regions, stream);
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation clear");
  if (q_tiles == 0) return PIC_OK;
  if ((long long)q_tiles * a.splits > 65535 || batch > 65535 || Hkv > 65535)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: grid too large");
  const dim3 grid((unsigned)(q_tiles * a.splits), Hkv, batch);
  if (D == 128) {
    const int smem = DLayout<128>::kAlloc;
    e = cudaFuncSetAttribute(deviation_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) deviation_kernel<128><<<grid, kThreads, smem, stream>>>(tq, tka, tkb, a);
  } else {
    const int smem = DLayout<64>::kAlloc;
    e = cudaFuncSetAttribute(deviation_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) deviation_kernel<64><<<grid, kThreads, smem, stream>>>(tq, tka, tkb, a);
  }
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation smem attribute");
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation launch");
  return PIC_OK;
}
