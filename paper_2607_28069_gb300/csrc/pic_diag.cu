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

// warp 0 TMA producer, warp 1 MMA issuer, warps 2-9 compute, warp 10 key regions
constexpr int kThreads = 352;
constexpr int kComputeWarps = 8;  // two per TMEM lane quarter, each on half the key columns
constexpr int kRegionWarp = 10;
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
  static constexpr int kTable = kBar + 256;  // document table, sized at launch
  // offsets and lengths int32 [max_docs] each, then the region bounds
  // int32 [max_docs][n_regions + 1]
  static size_t alloc(int max_docs, int n_regions) {
    return 1024 + kTable + (size_t)max_docs * 4 * (n_regions + 3);
  }
};

enum {
  DB_Q = 0,
  DB_KFULL = 1,
  DB_KEMPTY = DB_KFULL + NS,
  DB_SFULL = DB_KEMPTY + NS,  // per S buffer
  DB_SFREE = DB_SFULL + 2,    // per S buffer, one arrival per compute warp
  DB_RFULL = DB_SFREE + 2,    // per region buffer (the region bytes of a tile)
  DB_FINAL = DB_RFULL + 2,
  DB_COUNT = DB_FINAL + 1
};

struct DevArgs {
  int Hq, Hkv, G, max_inline, max_docs, max_ctx, R_pad, n_regions, splits;
  long long num_pages, layer_row0, oob_row;
  const int32_t *inline_pos, *inline_len, *query_len, *ids, *doc_len, *doc_offset;
  const int64_t *slots;
  const float *lse_a, *lse_b;
  double edges[kMaxRegions + 1];
  double *sums;
  unsigned long long *counts;
  int32_t *status;
  float scale_log2;
};

// The request's document table in shared memory: the documents' offsets
// ascend (canonical order), so the document holding a logical position t is
// the last one starting at or before t, and t - offset is its token index.
// doc_at: that document (0 when t precedes every document), by bisection.
__device__ int doc_at(const int32_t *s_off, int m, long long t) {
  int lo = 0, hi = m - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s_off[mid] <= t) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Regions of the keys at logical positions t .. t+3 (-1: not a document
// token, or in no region), packed one byte per key, searching forward from
// document k, which starts at or before t (or is document 0).  One document
// lookup serves the four keys unless the next document starts among them.
__device__ uint32_t four_regions(const int32_t *s_off, const int32_t *s_bnd, int m, int R1, int k,
                                 long long t) {
  if (m == 0) return 0xffffffffu;
  while (k + 1 < m && s_off[k + 1] <= t) ++k;
  long long off = s_off[k], nxt = k + 1 < m ? s_off[k + 1] : LLONG_MAX;
  int bd[kMaxRegions + 1];
#pragma unroll
  for (int i = 0; i <= kMaxRegions; ++i) bd[i] = i < R1 ? s_bnd[k * R1 + i] : 0;
  uint32_t packed = 0;
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const long long te = t + e;
    if (te >= nxt) {
      while (k + 1 < m && s_off[k + 1] <= te) ++k;
      off = s_off[k];
      nxt = k + 1 < m ? s_off[k + 1] : LLONG_MAX;
#pragma unroll
      for (int i = 0; i <= kMaxRegions; ++i) bd[i] = i < R1 ? s_bnd[k * R1 + i] : 0;
    }
    int reg = -1;
    const long long jj = te - off;  // negative before the first document
#pragma unroll
    for (int i = 0; i < kMaxRegions; ++i)
      if (i + 1 < R1 && jj >= bd[i] && jj < bd[i + 1]) reg = i;
    packed |= (uint32_t)(uint8_t)(int8_t)reg << (8 * e);
  }
  return packed;
}

// CTA = (128-row query tile, key split, kv head, request).  Per 128-key tile
// of the documents' span: the producer loads the tile of both caches (page
// boxes through the block layout, as the prefill attention does), one after
// the other, and the region warp writes the tile's key regions; the issuer
// computes [S_A S_B] = Q [K_A; K_B]^T, one N = 256 MMA per 16-deep slice,
// into a TMEM buffer (two buffers, so the next tile's MMAs overlap this
// one's exponentials); each compute thread owns one query row, reads both
// rows of scores from TMEM 32 columns at a time and adds |p_A - p_B| to its
// region.
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    deviation_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_ka,
                     const __grid_constant__ CUtensorMap tm_kb, DevArgs a) {
  using L = DLayout<D>;
  constexpr int PANELS = D / 64;
  constexpr uint32_t IDESC_QK = idesc_bf16(BM, 2 * BN, false, false);
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
    s_m = a.max_docs;
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

  // ---- the request's document table: offset, length and region bounds
  // ceil(e_i n) (double-precision products) of each document; the request's
  // documents end at the first doc_offset of -1
  const int R1 = a.n_regions + 1;
  int32_t *s_off = reinterpret_cast<int32_t *>(smem + L::kTable);
  int32_t *s_len = s_off + a.max_docs;
  int32_t *s_bnd = s_len + a.max_docs;
  for (int k = tid; k < a.max_docs; k += kThreads) {
    const int off = a.doc_offset[(size_t)b * a.max_docs + k];
    if (off < 0) {
      atomicMin(&s_m, k);
      continue;
    }
    const int id = a.ids[(size_t)b * a.max_docs + k];
    const int nk = id >= 0 ? a.doc_len[id] : 0;
    s_off[k] = off;
    s_len[k] = nk;
    for (int i = 0; i < R1; ++i) s_bnd[k * R1 + i] = (int)ceil(a.edges[i] * nk);
  }
  __syncthreads();

  // ---- the work of this CTA (uniform)
  const int tin = min(max(a.inline_len[b], 0), a.max_inline);
  const int tq = min(max(a.query_len[b], 0), tin);
  const int row_begin = (tin - tq) * a.G, row_end = tin * a.G;
  const int r0 = row_begin + qt * BM;
  const int m = s_m;
  long long key_lo = 0, key_hi = 0;
  if (m > 0) {
    key_lo = s_off[0];
    key_hi = (long long)s_off[m - 1] + s_len[m - 1];
  }
  const int kt0 = (int)(key_lo / BN);
  const int n_kt = key_hi > key_lo ? (int)((key_hi - 1) / BN) - kt0 + 1 : 0;
  const int per = (n_kt + a.splits - 1) / a.splits;
  const int kv_begin = split * per;
  const int n = max(0, min(per, n_kt - kv_begin));

  // the number of terms of each region: one CTA per request
  if (qt == 0 && split == 0 && hk == 0 && warp >= 2 && warp < 2 + kComputeWarps)
    for (int k = tid - 64; k < m; k += 32 * kComputeWarps)
      for (int i = 0; i < a.n_regions; ++i) {
        const long long lo = s_bnd[k * R1 + i], hi = s_bnd[k * R1 + i + 1];
        if (hi > lo)
          atomicAdd(&a.counts[(size_t)b * a.n_regions + i], (unsigned long long)(hi - lo) * tq * a.Hq);
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
      // lanes 0..7: the slot of the first position of page `lane` of tile
      // jj, loaded one tile ahead so that the TMA issue never waits on it
      auto load_slot = [&](int jj) -> long long {
        if (lane >= 8 || jj >= n) return -1;
        const long long t = ((long long)(kt0 + kv_begin + jj) * 8 + lane) * 16;
        return t < a.max_ctx ? a.slots[(size_t)b * a.max_ctx + t] : -1;
      };
      long long slot_next = load_slot(0);
      for (int j = 0; j < n; ++j) {
        const int st = j % NS;
        const long long slot = slot_next;
        slot_next = load_slot(j + 1);
        int y = (int)a.oob_row;  // lanes 0..7: page row of page `lane` of the tile
        if (slot >= 0 && (slot >> 4) < a.num_pages)
          y = (int)(a.layer_row0 + ((slot >> 4) * a.Hkv + hk) * 16);
        bool ok = true;
        if (j >= NS) ok = mbar_wait(bar(DB_KEMPTY + st), ((j / NS) - 1) & 1, abort_flag, a.status, b);
        if (!__all_sync(0xffffffffu, ok)) break;
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
    } else if (warp == kRegionWarp) {
      // ================================================ key regions
      // Lane l writes the regions of keys 4l .. 4l+3 of each tile; the bytes
      // go where tile j - 2's were, once its scores are consumed.
      int kc = m > 0 ? doc_at(s_off, m, (long long)(kt0 + kv_begin) * BN) : 0;
      for (int j = 0; j < n; ++j) {
        const long long t0 = (long long)(kt0 + kv_begin + j) * BN;
        const uint32_t packed = four_regions(s_off, s_bnd, m, R1, kc, t0 + 4 * lane);
        while (kc + 1 < m && s_off[kc + 1] <= t0 + BN) ++kc;
        bool ok = true;
        if (j >= 2) ok = mbar_wait(bar(DB_SFREE + (j & 1)), ((j >> 1) - 1) & 1, abort_flag, a.status, b);
        if (!__all_sync(0xffffffffu, ok)) break;
        reinterpret_cast<uint32_t *>(s_reg + (j & 1) * BN)[lane] = packed;
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(DB_RFULL + (j & 1)));
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
          // K_B's tile follows K_A's with the same 8-row group stride, so
          // one 256-row operand covers both: S_A in columns 0..127 of the
          // buffer, S_B in 128..255
          const uint32_t tS = tbase + buf * 256;
          const uint64_t dk = dK + (uint64_t)((st * 2 * L::kTile) >> 4);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t qd = dQ + ((kk >> 2) * (BM * 128) + (kk & 3) * 32) / 16;
            const uint64_t ko = ((kk >> 2) * kPanelOff + (kk & 3) * 32) / 16;
            mma_ss(tS, qd, dk + ko, IDESC_QK, kk > 0);
          }
          mma_commit(bar(DB_SFULL + buf));
          mma_commit(bar(DB_KEMPTY + st));
        }
        mma_commit(bar(DB_FINAL));
      }
    } else {
      // ================================================ compute warps
      // Two warps per TMEM lane quarter, each on 64 of the 128 key columns,
      // 32 at a time.  The 32 terms of a chunk are computed without branches
      // (the exponentials pipeline); a chunk whose keys all lie in one region
      // (the region bytes are the same for every row) is summed at once, one
      // in no region is skipped, and only a chunk across a region or
      // document boundary is summed key by key.  A key after a row's
      // position (an inline span taken as a query row before a later
      // document) has p_A = p_B = 0.
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
      const uint32_t tl = tbase + ((uint32_t)(wq * 32) << 16) + half * 64;
      float acc[kMaxRegions];
#pragma unroll
      for (int i = 0; i < kMaxRegions; ++i) acc[i] = 0.f;
      auto add_to = [&](int reg, float v) {
#pragma unroll
        for (int i = 0; i < kMaxRegions; ++i)
          if (i == reg) acc[i] += v;
      };
      for (int j = 0; j < n; ++j) {
        const int buf = j & 1;
        // the region bytes of tile j written, S(j) ready
        bool ok = mbar_wait(bar(DB_RFULL + buf), (j >> 1) & 1, abort_flag, a.status, b);
        if (ok) ok = mbar_wait(bar(DB_SFULL + buf), (j >> 1) & 1, abort_flag, a.status, b);
        if (!__all_sync(0xffffffffu, ok)) break;
        tc_fence_after();
#pragma unroll 1
        for (int c0 = 0; c0 < 64; c0 += 32) {
          const int8_t *rr = s_reg + buf * BN + half * 64 + c0;
          const uint4 w0 = *reinterpret_cast<const uint4 *>(rr);
          const uint4 w1 = *reinterpret_cast<const uint4 *>(rr + 16);
          const int reg0 = rr[0];
          const uint32_t rep = (uint32_t)(uint8_t)rr[0] * 0x01010101u;
          const bool uniform = w0.x == rep && w0.y == rep && w0.z == rep && w0.w == rep &&
                               w1.x == rep && w1.y == rep && w1.z == rep && w1.w == rep;
          if (uniform && reg0 < 0) continue;  // no key of the chunk is in a region
          float sa[32], sb[32];
          tmem_ld32(tl + buf * 256 + c0, reinterpret_cast<uint32_t *>(sa));
          tmem_ld32(tl + buf * 256 + 128 + c0, reinterpret_cast<uint32_t *>(sb));
          tmem_wait_ld();
          // keys 0..lim of the chunk are at or before this row's position
          const long long t0 = (long long)(kt0 + kv_begin + j) * BN + half * 64 + c0;
          const int lim = (int)min(max(qpos - t0, -1ll), 31ll);
          if (uniform && __all_sync(0xffffffffu, lim == 31)) {
            // one region, every key visible to every row of the warp: six
            // instructions a term (two FFMA, two EX2, two FADD)
            float v0 = 0.f, v1 = 0.f, v2 = 0.f, v3 = 0.f;
#pragma unroll
            for (int c = 0; c < 32; c += 4) {
              v0 += fabsf(ex2(fmaf(sa[c], a.scale_log2, -la)) - ex2(fmaf(sb[c], a.scale_log2, -lb)));
              v1 += fabsf(ex2(fmaf(sa[c + 1], a.scale_log2, -la)) - ex2(fmaf(sb[c + 1], a.scale_log2, -lb)));
              v2 += fabsf(ex2(fmaf(sa[c + 2], a.scale_log2, -la)) - ex2(fmaf(sb[c + 2], a.scale_log2, -lb)));
              v3 += fabsf(ex2(fmaf(sa[c + 3], a.scale_log2, -la)) - ex2(fmaf(sb[c + 3], a.scale_log2, -lb)));
            }
            add_to(reg0, (v0 + v1) + (v2 + v3));
          } else {
            // a region or document boundary inside the chunk, or keys after
            // some row's position: the masked terms first, then one masked
            // sum per region, with no branch between the terms (a branch per
            // key would serialise the exponentials)
#pragma unroll
            for (int c = 0; c < 32; ++c) {
              const float d = fabsf(ex2(fmaf(sa[c], a.scale_log2, -la)) - ex2(fmaf(sb[c], a.scale_log2, -lb)));
              sa[c] = c <= lim ? d : 0.f;
            }
            int rg[32];
#pragma unroll
            for (int c = 0; c < 32; ++c) rg[c] = rr[c];
#pragma unroll 1
            for (int i = 0; i < a.n_regions; ++i) {
              float v0 = 0.f, v1 = 0.f;
#pragma unroll
              for (int c = 0; c < 32; c += 2) {
                v0 += rg[c] == i ? sa[c] : 0.f;
                v1 += rg[c + 1] == i ? sa[c + 1] : 0.f;
              }
              add_to(i, v0 + v1);
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(DB_SFREE + buf));
      }
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
    const int32_t *doc_offset, const int64_t *slot_mapping,
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
      !slot_mapping || !k_cache_a || !k_cache_b || !lse_a || !lse_b || !workspace ||
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
  a.lse_a = lse_a;
  a.lse_b = lse_b;
  for (int i = 0; i <= kMaxRegions; ++i) a.edges[i] = i <= n_regions ? edges[i] : 1.0;
  a.sums = sums;
  a.counts = reinterpret_cast<unsigned long long *>(counts);
  a.status = status;
  a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D));
  // query tiles: the query rows of a request are its last query_len inline
  // tokens times G.  Key splits (every split adds its own partial sums): one
  // CTA per SM, so a launch takes ceil(CTAs / 152) rounds of one CTA's key
  // tiles plus about two tiles of pipeline fill; take the split count that
  // minimises that
  const int q_tiles = (int)(((long long)max_query_len * G + BM - 1) / BM);
  const int kt_max = (max_ctx + BN - 1) / BN;
  const long long groups = (long long)batch * Hkv * std::max(q_tiles, 1);
  a.splits = 1;
  long long best = -1;
  for (int sp = 1; sp <= std::min(kt_max, 64); ++sp) {
    const long long cost = ((groups * sp + 151) / 152) * ((kt_max + sp - 1) / sp + 2);
    if (best < 0 || cost < best) best = cost, a.splits = sp;
  }
  cudaError_t e = cudaMemsetAsync(sums, 0, sizeof(double) * batch * n_regions, stream);
  if (e == cudaSuccess) e = cudaMemsetAsync(counts, 0, sizeof(int64_t) * batch * n_regions, stream);
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation clear");
  if (q_tiles == 0) return PIC_OK;
  if ((long long)q_tiles * a.splits > 65535 || batch > 65535 || Hkv > 65535)
    return fail(PIC_ERR_INVALID_ARG, "pic_attention_deviation: grid too large");
  const dim3 grid((unsigned)(q_tiles * a.splits), Hkv, batch);
  const size_t smem_need = D == 128 ? DLayout<128>::alloc(max_docs, n_regions)
                                     : DLayout<64>::alloc(max_docs, n_regions);
  if (smem_need > 227 * 1024)
    return fail(PIC_ERR_UNSUPPORTED, "pic_attention_deviation: %d documents per request do not fit the "
                "shared-memory document table", max_docs);
  if (D == 128) {
    const int smem = (int)smem_need;
    e = cudaFuncSetAttribute(deviation_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) deviation_kernel<128><<<grid, kThreads, smem, stream>>>(tq, tka, tkb, a);
  } else {
    const int smem = (int)smem_need;
    e = cudaFuncSetAttribute(deviation_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess) deviation_kernel<64><<<grid, kThreads, smem, stream>>>(tq, tka, tkb, a);
  }
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation smem attribute");
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_attention_deviation launch");
  return PIC_OK;
}
