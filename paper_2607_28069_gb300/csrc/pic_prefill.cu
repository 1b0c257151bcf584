// pic_attend_prefill: inline-token prefill over the stitched cache.
//
// SemPIC, "Cache-hit serving": a cache hit processes only the request-specific
// inline tokens through the unchanged decoder; appendix "Position-Independent
// Linking": inline KVs are interleaved with the prepared document states and a
// frontier causal mask keeps every inline token from seeing logical
// successors.  The Reader is the frozen base model (Eq. 7), so its attention is
// ordinary GQA softmax attention with scale 1/sqrt(d).
//
// pic_append_inline (one layer, one launch): append_kernel applies RoPE to
//     each inline key at its logical position and writes it with its value
//     to the paged cache, and writes the rotated queries into a GQA-packed
//     workspace [B][Hkv][rows][d] whose row r of kv head g is query head
//     g*G + r % G of inline token r / G.  One 128-row tile therefore holds
//     every query head that shares a K/V tile.
// pic_attend_prefill (one layer):
//  1. attn_kernel: one CTA per (128-row query tile, key split, kv head,
//     request).  Warp-specialised: warp 0 issues TMA loads (Q once, then
//     128-key K and V tiles page by page from the paged cache through the
//     block table, 3-stage ring; its 32 lanes issue the 32 page boxes of a
//     tile at once and fetch the next tile's block-table entries ahead), warp 1 issues tcgen05.mma (S = Q K^T into
//     TMEM, then O += P V with P read from TMEM), warps 2-5 run the online
//     softmax on S rows straight from TMEM (one thread per row), write P back
//     to TMEM as bf16 over S, rescale O only when the running maximum grew by
//     more than 2^8, and finally normalise O.  Scores are kept in the log2
//     domain (scale folded with log2 e) and exponentiated with ex2.approx.
//  2. combine_kernel (only when the key range of a tile is split over several
//     CTAs): log-sum-exp merge of the per-split partials (O, m, l), one warp
//     per query row.
#include <algorithm>
#include <functional>
#include <vector>

#include "pic_internal.cuh"

namespace pic {
namespace prefill {

constexpr int BM = 128;  // query rows per tile (TMEM lanes)
constexpr int NQ = 2;    // query tiles per CTA, sharing every K/V tile
constexpr int BN = 128;  // keys per KV tile
constexpr int NSK = 3;   // K ring stages (released after the last QK of a tile)
constexpr int NSV = 2;   // V ring stages (released after the last PV of a tile)
constexpr int kThreads = 128 + NQ * 128;  // K producer, MMA, NQ softmax warpgroups, V producer, relay
// Rotate-on-load adds a warpgroup that rotates the document keys of each K
// tile (warps 12-15); its roles are warpgroup-aligned so the registers can be
// redistributed with setmaxnreg: the control warpgroup (K producer, MMA, V
// producer, relay) and the rotators give registers to the softmax warpgroups.
constexpr int kThreadsFused = 512;
constexpr int kRegLaunchFused = 65536 / kThreadsFused;  // 128 per thread at launch
constexpr int kRegCtl = 88, kRegRot = 72, kRegSoftmax = 176;
static_assert(128 * kRegCtl + 128 * kRegRot + 256 * kRegSoftmax <= 128 * 4 * kRegLaunchFused,
              "setmaxnreg split exceeds the registers the CTA is launched with");
template <bool kFused>
constexpr int threads_of() { return kFused ? kThreadsFused : kThreads; }
constexpr int kWarpV = 2 + 4 * NQ;        // the V producer warp
constexpr int kWarpRelay = kWarpV + 1;    // waits on behalf of the MMA issuer
// Named barriers between the relay warp and the MMA warp (64 threads each);
// 0 is __syncthreads, 1 and 2 belong to the softmax warpgroups' epilogue.
constexpr int kNbPv = 3;  // + t: P_t(j-1) and V(j-1) are ready
constexpr int kNbK = 5;   // K(j) is ready
constexpr int kMaxSplits = 32;
constexpr uint32_t kTmemCols = 512;

template <int D>
struct Layout {
  static constexpr int kTile = BN * D * 2;  // bytes of one K or V tile
  static constexpr int kQTile = BM * D * 2;
  static constexpr int kQ = 0;
  static constexpr int kK = kQ + NQ * kQTile;
  static constexpr int kV = kK + NSK * kTile;
  static constexpr int kBar = kV + NSV * kTile;
  // rotate-on-load: per K stage the sources of its 8 pages ({kind, delta}),
  // and for pages across a boundary each row's document (-1: inline)
  static constexpr int kInfo = kBar + 256;
  static constexpr int kRowDoc = kInfo + NSK * 8 * 8;
  static constexpr int kBytes = kRowDoc + NSK * 8 * 16 * 2;
  static constexpr int kAlloc = kBytes + 1024;  // slack for 1024-byte alignment
};

// mbarrier slots (8 bytes each) inside the barrier area
enum {
  B_Q = 0,
  B_KFULL = 1,
  B_KEMPTY = B_KFULL + NSK,
  B_VFULL = B_KEMPTY + NSK,
  B_VEMPTY = B_VFULL + NSV,
  B_SFULL = B_VEMPTY + NSV,  // one per query tile
  B_PFULL = B_SFULL + NQ,     // one per query tile (one arrival per softmax warp)
  B_OFINAL = B_PFULL + NQ,
  B_KROT = B_OFINAL + 1,  // rotate-on-load: this CTA's half of K(j) rotated (one arrival per rotator warp)
  B_KPEER = B_KROT + NSK,  // rotate-on-load: the cluster peer's rotated half of K(j) has landed
  B_EXIT = B_KPEER + NSK,  // rotate-on-load: the peer is done with this CTA's shared memory
  B_COUNT = B_EXIT + 1
};

struct Params {
  int batch, Hq, Hkv, G, max_inline, R_pad, m_tiles, num_splits, max_pages, oob_row;
  long long num_pages, layer_row0;
  const int32_t *inline_pos, *inline_len, *block_table;
  __nv_bfloat16 *out;
  float *lse, *part_ml;
  __half *part_o;  // split partials: O / l per row, fp16
  int32_t *status;
  float scale_log2;
};

// Source of one page of 16 positions (written by fused_setup_kernel): kind as
// PageSrc below; for kind 1 the pool row of its first position and the
// document's index k in the request (field `delta`).
struct alignas(16) PageSrcEntry {
  int32_t kind, delta;
  int64_t row;
};

// Rotate-on-load sources (attn_kernel<D, true>): every logical position's
// source from pic_compose's token map -- a pool row of a document (moved by
// that document's delta) or, for inline tokens, the paged cache.
struct FusedArgs {
  const int64_t *tok_map;    // [batch][max_ctx]: (k << 40) | pool row, -1 inline
  const int32_t *doc_delta;  // [batch][max_docs]
  const __nv_bfloat16 *k_pool, *v_pool;    // [L][pool_tokens][Hkv][D]
  const __nv_bfloat16 *k_cache, *v_cache;  // [L][num_pages][Hkv][16][D]
  long long pool_tokens;
  int max_ctx, max_docs, layer;
  bool pool_boxes;  // false: the pool is too small for a page box (all pages row by row)
  const PageSrcEntry *page_src;  // [batch][n_pidx]
  const float2 *doc_cs;          // [batch][max_docs][D/2]: cos/sin of each document's delta
  int n_pidx, half;
};

// Byte offset of the 16-byte piece ch (0 .. D/8-1) of row r (0..15) of a page
// inside a K/V ring tile, as the page boxes lay it out with the 128-byte
// swizzle: [8-row half][64-column panel][8 rows][128 B] at d = 128,
// [16 rows][128 B] at d = 64.
template <int D>
PIC_DEV uint32_t page_piece(int r, int ch) {
  const int c8 = ch & 7;
  if constexpr (D == 128)
    return (uint32_t)((r >> 3) * 2048 + (ch >> 3) * 1024 + (r & 7) * 128 + ((c8 ^ (r & 7)) << 4));
  else
    return (uint32_t)(r * 128 + ((c8 ^ (r & 7)) << 4));
}

// Set-up of a rotate-on-load call (one launch, ahead of the attention):
// blocks [0, page_blocks) write the source of every page of positions
// < max_ctx of every request, from the token map -- a page whose first and
// last positions are rows of one document is that document's (documents
// occupy contiguous positions), a page of inline tokens only is the cache's,
// anything else is mixed -- one warp per page; blocks from page_blocks on
// write cos/sin of delta_k * theta_i for every listed document k, as
// pic_relocate forms them (fp64-reduced angle; the fast sine and cosine with
// per-layer tables, as pic_relocate's per-layer instantiation).
__global__ void __launch_bounds__(256) fused_setup_kernel(FusedArgs f, RopeParams rp, int batch,
                                                          int page_blocks, int32_t *status) {
  pdl_entry();
  const int b = blockIdx.y;
  if (b >= batch) return;
  if ((int)blockIdx.x >= page_blocks) {
    const int k0 = ((int)blockIdx.x - page_blocks) * (256 / f.half);
    const int k = k0 + (int)threadIdx.x / f.half, i = (int)threadIdx.x % f.half;
    if (k >= f.max_docs || (int)threadIdx.x >= (256 / f.half) * f.half) return;
    const int delta = f.doc_delta[(size_t)b * f.max_docs + k];
    const double th = rope_theta(rp, f.layer, i);
    const_cast<float2 *>(f.doc_cs)[((size_t)b * f.max_docs + k) * f.half + i] =
        rp.layer_theta ? rope_cos_sin_fast(delta, th) : rope_cos_sin(delta, th);
    return;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long pidx = (long long)blockIdx.x * 8 + warp;
  if (pidx >= f.n_pidx) return;
  const long long t = pidx * 16 + (lane & 15);
  const long long tm = t < f.max_ctx ? f.tok_map[(size_t)b * f.max_ctx + t] : -1;
  const unsigned inl = __ballot_sync(0xffffffffu, tm < 0) & 0xffffu;
  const long long first = __shfl_sync(0xffffffffu, tm, 0), last = __shfl_sync(0xffffffffu, tm, 15);
  if (lane != 0) return;
  PageSrcEntry e;
  e.kind = inl == 0xffffu ? 0 : 2;
  e.delta = 0;
  e.row = 0;
  if (e.kind == 2 && f.pool_boxes && first >= 0 && last >= 0 && (first >> 40) == (last >> 40)) {
    const int k = (int)(first >> 40);
    const long long row = first & ((1LL << 40) - 1);
    if (k < f.max_docs && row + 15 < f.pool_tokens) {
      e.kind = 1;
      e.delta = k;  // the document index: its cos/sin are row k of doc_cs
      e.row = row;
    } else {
      dev_fail(status, PIC_DEV_BAD_DOC_LEN, b);
    }
  }
  const_cast<PageSrcEntry *>(f.page_src)[(size_t)b * f.n_pidx + pidx] = e;
}

// Sources of the 8 pages of a key tile (one page per lane 0..7).
struct PageSrc {
  int kind;   // 0: inline tokens (cache box at row y), 1: one document's rows
              // (pool box at row y, rotated by delta), 2: mixed (row by row;
              // y = the page's cache rows for its inline tokens)
  int y, delta;
};

// One CTA = (pair of 128-row query tiles, key split, kv head, request).
// TMEM: S_t at columns 128 t (P_t written over it as bf16), O_t at 256 + 128 t.
// MMA order per KV tile j: PV_0(j-1), QK_0(j), PV_1(j-1), QK_1(j).  Because
// tcgen05 MMAs of one thread complete in order, "S_t(j) is ready" implies
// PV_t(j-1) has finished, so softmax t may rescale O_t right away, and
// softmax 0 runs while the tensor core works on tile 1 and vice versa.
// The MMA issuer does no mbarrier wait inside its loop: an mbarrier wait of
// a thread queues behind the MMAs that thread issued, so each one left the
// tensor core idle for a while.  A relay warp waits for K(j), V(j-1) and
// P_t(j-1) in the issuer's order and hands each over on a named barrier.
//
// kFused (rotate-on-load, pic_attend_prefill_fused): the key and value tiles
// are assembled from the document pool and the cache instead of the stitched
// cache alone.  A page whose 16 positions are all one document's comes from
// the pool as one box (the document's rows are consecutive there); a page of
// inline tokens from the cache as before; a page across a boundary is filled
// row by row by the producer warp.  A rotator warpgroup then rotates every
// document row in shared memory by its document's delta -- the same fp32
// arithmetic and bf16 rounding as the relocation, so the tile holds exactly
// the keys pic_relocate would have stitched.  The CTAs run in clusters of
// two (two query pairs of one key split): each loads and rotates half of
// every key tile and bulk-copies the rotated pages into the other's ring, so
// K(j) is complete when its own half is rotated (B_KROT) and the peer's half
// has landed (B_KPEER); the QK commits are multicast to both CTAs' B_KEMPTY.
// Everything downstream (MMAs, softmax, merge) is the materialised kernel's.
//
// The body is one function per group of warps (kGroup: 0 the control
// warpgroup, 1 the rotators, 2 the softmax warpgroups; -1 all warps of the
// materialised kernel), entered right after the group's setmaxnreg, so no
// value is live across the register reallocation (values live across it
// were spilled and reloaded in the control warps' loops).
template <int D, bool kFused, int kGroup>
__device__ __forceinline__ void attn_body(const CUtensorMap &tm_q, const CUtensorMap &tm_k,
                                          const CUtensorMap &tm_v, const CUtensorMap &tm_kp,
                                          const CUtensorMap &tm_vp, Params p, FusedArgs f,
                                          RopeParams rp) {
  using L = Layout<D>;
  constexpr int PANELS = D / 64;
  constexpr uint32_t IDESC_QK = idesc_bf16(BM, BN, false, false);
  constexpr uint32_t IDESC_PV = idesc_bf16(BM, D, false, true);
  // K/V ring tiles are page-major: page p of a tile at p * kPageBytes.  At
  // d = 128 a page lands as [8-row half][64-column panel][8 rows][128 B]
  // (8-row groups 2048 B apart, panels 1024 B apart); at d = 64 as
  // [16 rows][128 B] (groups 1024 B apart, one panel).
  constexpr uint32_t kPageBytes = 16 * D * 2;
  constexpr uint32_t kGroupStride = PANELS == 2 ? 2048 : 1024;
  constexpr uint32_t kPanelOff = PANELS == 2 ? 1024 : BN * 128;

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + L::kBar;
  auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + L::kBar + 8 * B_COUNT);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::kBar + 8 * B_COUNT + 8);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // Warp roles: 0 K producer, 1 MMA issuer, then either 2-9 softmax, 10 V
  // producer, 11 relay, or (rotate-on-load) 2 V producer, 3 relay, 4-11
  // softmax, 12-15 rotators.
  constexpr int W_V = kFused ? 2 : kWarpV;
  constexpr int W_RELAY = kFused ? 3 : kWarpRelay;
  constexpr int W_SM = kFused ? 4 : 2;  // first softmax warp
  constexpr int W_ROT = 12;             // first rotator warp (rotate-on-load)
  // Grid (pair + npairs * split, kv head, request).  CTAs start in linear
  // block order: the query pairs that read one key split of one (request,
  // kv head) are adjacent, so they start in the same wave and read each K/V
  // tile within a short window (from DRAM once, then from L2); a split-minor
  // order let waves cut through those sets and the late readers of a range
  // found it evicted (1.48x the algorithmic K/V read on the 4 x 139k
  // workload, 1.05x in this order).  Query tiles are counted from a
  // request's last row, so pair 0, which sees the most keys, goes first.
  const int npairs = (int)gridDim.x / p.num_splits;
  const int split = (int)blockIdx.x / npairs;
  const int pair = (int)blockIdx.x % npairs;
  const int hk = blockIdx.y, b = blockIdx.z;
  const int detail = b;

  // ---- set-up that reads nothing the previous kernel writes: it runs before
  // the programmatic-launch wait, while that kernel may still be finishing
  if (threadIdx.x == 0) {
    for (int i = 0; i < B_COUNT; ++i)
      mbar_init(bar(i), ((i >= B_PFULL && i < B_PFULL + NQ) || (i >= B_KROT && i < B_KROT + NSK))
                            ? 4
                        : (kFused && i >= B_KEMPTY && i < B_KEMPTY + NSK) ? 2  // both CTAs' QK
                                                                          : 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_q);
    prefetch_tmap(&tm_k);
    prefetch_tmap(&tm_v);
    if constexpr (kFused) {
      prefetch_tmap(&tm_kp);
      prefetch_tmap(&tm_vp);
    }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // rotate-on-load runs in clusters of two CTAs (consecutive query pairs of
  // one key split): each loads and rotates half of every key tile and copies
  // it into the other's ring, so the barriers must be initialised in both
  // before either touches the other's
  const uint32_t crank = kFused ? cluster_rank() : 0u, cpeer = crank ^ 1u;
  if constexpr (kFused) cluster_sync_all();
  const uint32_t tbase = *tmem_slot;
  asm volatile("griddepcontrol.wait;" ::: "memory");  // the kernel before has finished
  auto release_and_exit = [&]() {  // a CTA without work frees its TMEM
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tbase, kTmemCols);
    }
  };

  // ---- work of this CTA (uniform across threads)
  const int tin = min(max(p.inline_len[b], 0), p.max_inline);
  const int rows = tin * p.G;
  const int32_t *ipos = p.inline_pos + (size_t)b * p.max_inline;
  // Query tile mt of a request holds its packed rows [rows - 128 (mt + 1),
  // rows - 128 mt): the tiles are aligned to the request's last row, so a
  // query chunk whose rows are a multiple of 128 fills whole tiles and never
  // shares one with the prefix rows, which see only the prefix keys.  The
  // lowest tile may start below row 0 (those rows are padding: loaded from
  // outside the request, fully masked, never written).  Tile t of the pair is
  // mt = NQ pair + t, so tile 0 has the most keys and tile 1 at most as many.
  int r0[NQ], kmin[NQ], kmax[NQ], ntile = 0;
#pragma unroll
  for (int t = 0; t < NQ; ++t) {
    const int mt = pair * NQ + t;
    r0[t] = rows - (mt + 1) * BM;
    kmin[t] = kmax[t] = -1;
    if (mt < p.m_tiles && r0[t] + BM > 0) {
      kmin[t] = ipos[max(r0[t], 0) / p.G];
      kmax[t] = ipos[(r0[t] + BM - 1) / p.G];
      ntile = t + 1;
    }
  }
  int kmax_all = kmax[0];
  if constexpr (kFused) {
    // Both CTAs of a cluster stream the key tiles of its upper pair, whose
    // first tile sees the most keys; the lower pair may have no rows and then
    // only loads, rotates and passes on its half of every key tile.
    const int mt_top = (pair & ~1) * NQ, r_top = rows - (mt_top + 1) * BM;
    kmax_all = (mt_top < p.m_tiles && r_top + BM > 0) ? ipos[(r_top + BM - 1) / p.G] : -1;
    if (kmax_all < 0) {  // neither pair of the cluster has a query row
      release_and_exit();
      return;
    }
  } else if (ntile == 0) {  // no query row in this pair
    release_and_exit();
    return;
  }
  const int n_kv_all = kmax_all >= 0 ? kmax_all / BN + 1 : 0;
  const int per = (n_kv_all + p.num_splits - 1) / p.num_splits;
  const int kv_begin = split * per;
  const int n = max(0, min(per, n_kv_all - kv_begin));
  int nt[NQ];  // KV tiles of this split that query tile t needs
#pragma unroll
  for (int t = 0; t < NQ; ++t)
    nt[t] = (t < ntile && kmax[t] >= 0) ? max(0, min(n, kmax[t] / BN + 1 - kv_begin)) : 0;
  auto part_row0 = [&](int t) {
    return ((((size_t)b * p.Hkv + hk) * p.m_tiles + pair * NQ + t) * p.num_splits + split) * BM;
  };

  if (n == 0) {  // empty split: neutral partial state for every tile
    if (p.num_splits > 1 && threadIdx.x < BM)
#pragma unroll
      for (int t = 0; t < NQ; ++t) {
        if (t >= ntile) break;
        p.part_ml[(part_row0(t) + threadIdx.x) * 2] = -INFINITY;
        p.part_ml[(part_row0(t) + threadIdx.x) * 2 + 1] = 0.f;
      }
    release_and_exit();
    return;
  }

  // ---- the roles, each a lambda called by the warps that take it
  auto role_producer = [&]() {
    // ===================================================== TMA producers
    // Warp 0 streams K tiles into a 3-deep ring, warp kWarpV V tiles into a
    // 2-deep ring.  Lane l < 8 moves page l of the tile as one box (a whole
    // page-head: 4 KB at d = 128, 2 KB at d = 64) and looks up the next
    // tile's block-table entry one iteration ahead.
    const bool is_k = warp == 0;
    const int nst = is_k ? NSK : NSV;
    const int b_full = is_k ? B_KFULL : B_VFULL, b_empty = is_k ? B_KEMPTY : B_VEMPTY;
    const uint32_t ring = sbase + (is_k ? L::kK : L::kV);
    const CUtensorMap *tmap = is_k ? &tm_k : &tm_v;
    const int32_t *bt = p.block_table + (size_t)b * p.max_pages;
    auto page_row = [&](int kt) -> int {  // lanes 0..7: TMA row of page `lane` of tile kt
      int y = p.oob_row;
      const int pidx = kt * 8 + lane;
      if (lane < 8 && pidx * 16 <= kmax_all && pidx < p.max_pages) {
        const int page = bt[pidx];
        if (page >= 0 && page < p.num_pages)
          y = (int)(p.layer_row0 + ((long long)page * p.Hkv + hk) * 16);
        else if (is_k)
          dev_fail(p.status, PIC_DEV_BAD_PAGE, detail);
      }
      return y;
    };
    if (is_k && lane == 0) {
      prefetch_tmap(&tm_q);
      prefetch_tmap(&tm_k);
      mbar_expect_tx(bar(B_Q), ntile * L::kQTile);
#pragma unroll
      for (int t = 0; t < NQ; ++t) {
        if (t >= ntile) break;
        const int qrow = (b * p.Hkv + hk) * p.R_pad + r0[t];
#pragma unroll
        for (int pn = 0; pn < PANELS; ++pn)
          tma_load_2d(sbase + L::kQ + t * L::kQTile + pn * BM * 128, &tm_q, pn * 64, qrow, bar(B_Q));
      }
    }
    if (!is_k && lane == 0) prefetch_tmap(&tm_v);
    if constexpr (!kFused) {
      int y_next = page_row(kv_begin);
      int issued = 0;
      for (int j = 0; j < n; ++j) {
        const int st = j % nst;
        const int y_mine = y_next;
        if (j + 1 < n) y_next = page_row(kv_begin + j + 1);
        if (j >= nst) {
          const bool ok = mbar_wait(bar(b_empty + st), ((j / nst) - 1) & 1, abort_flag, p.status, detail);
          if (!__all_sync(0xffffffffu, ok)) break;
        }
        if (lane == 0) mbar_expect_tx(bar(b_full + st), L::kTile);
        __syncwarp();
        if (lane < 8) {  // one box per page-head
          const uint32_t dst = ring + st * L::kTile + lane * kPageBytes;
          if constexpr (PANELS == 2)
            tma_load_4d(dst, tmap, 0, 0, 0, y_mine >> 3, bar(b_full + st));
          else
            tma_load_2d(dst, tmap, 0, y_mine, bar(b_full + st));
        }
        issued = j + 1;
      }
      if (lane == 0 && *abort_flag) {
        // Let the copies already issued land before the CTA exits.
        for (int j = max(0, issued - nst); j < issued; ++j)
          mbar_wait(bar(b_full + j % nst), (j / nst) & 1, abort_flag, p.status, detail);
      }
    } else {
      // ---- rotate-on-load producers: pages from the pool or the cache as the
      // page-source table says; mixed pages row by row.  The rotators (warps
      // 12-15) then rotate the K tile's document rows.
      const CUtensorMap *pmap = is_k ? &tm_kp : &tm_vp;
      if (lane == 0) prefetch_tmap(pmap);
      const int64_t *tmr = f.tok_map + (size_t)b * f.max_ctx;
      const __nv_bfloat16 *pool = is_k ? f.k_pool : f.v_pool;
      const __nv_bfloat16 *cache = is_k ? f.k_cache : f.v_cache;
      const PageSrcEntry *ps = f.page_src + (size_t)b * f.n_pidx;
      // lanes 0..7: the source of page `lane` of tile kt (kind 0 and 2 carry
      // the page's cache row, kind 1 the pool row)
      auto source = [&](int kt) -> PageSrc {
        PageSrc src{0, page_row(kt), 0};
        const int pidx = kt * 8 + lane;
        if (lane < 8 && pidx < f.n_pidx) {
          const PageSrcEntry e = ps[pidx];
          src.kind = e.kind;
          src.delta = e.delta;
          if (e.kind == 1) src.y = (int)((long long)f.layer * f.pool_tokens + e.row);
        }
        return src;
      };
      // The K producer fills its CTA's half of every key tile (pages
      // 4 crank .. 4 crank + 3; the cluster peer sends the rotated other
      // half), the V producer whole tiles.
      const bool mine = lane < 8 && (!is_k || (uint32_t)(lane >> 2) == crank);
      auto issue = [&](int st, int kt, const PageSrc &src) {
        const uint32_t stage = ring + st * L::kTile;
        const unsigned box_mask = __ballot_sync(0xffffffffu, mine && src.kind != 2);
        unsigned mixed = __ballot_sync(0xffffffffu, mine && src.kind == 2);
        if (lane == 0) {
          mbar_expect_tx_only(bar(b_full + st), __popc(box_mask) * kPageBytes);
          if (is_k) mbar_expect_tx(bar(B_KPEER + st), 4 * kPageBytes);
        }
        __syncwarp();
        if (mine && src.kind != 2) {
          const uint32_t dst = stage + lane * kPageBytes;
          if (src.kind == 0) {
            if constexpr (PANELS == 2)
              tma_load_4d(dst, tmap, 0, 0, 0, src.y >> 3, bar(b_full + st));
            else
              tma_load_2d(dst, tmap, 0, src.y, bar(b_full + st));
          } else {
            if constexpr (PANELS == 2)
              tma_load_5d(dst, pmap, 0, src.y, 0, 0, hk, bar(b_full + st));
            else
              tma_load_3d(dst, pmap, 0, hk, src.y, bar(b_full + st));
          }
        }
        while (mixed) {  // row by row: 16-byte loads, swizzled 16-byte stores
          const int q = __ffs(mixed) - 1;
          mixed &= mixed - 1;
          const int yq = __shfl_sync(0xffffffffu, src.y, q);
          // the page's 16 token-map entries (lane r < 16 holds row r's), then
          // every 16-byte piece of the page loaded at once, then stored
          const long long t_l = (long long)kt * BN + q * 16 + (lane & 15);
          const long long tv_l = t_l < f.max_ctx ? tmr[t_l] : -1;
          if (is_k && lane < 16)  // each row's document for the rotators (-1: inline)
            reinterpret_cast<int16_t *>(smem + L::kRowDoc)[(st * 8 + q) * 16 + lane] =
                (tv_l >= 0 && (tv_l >> 40) < f.max_docs) ? (int16_t)(tv_l >> 40) : (int16_t)-1;
          constexpr int CH = D / 8, PER = 16 * CH / 32, GRP = 4;  // GRP loads in flight per lane
#pragma unroll
          for (int i0 = 0; i0 < PER; i0 += GRP) {
            uint4 v[GRP];
#pragma unroll
            for (int i = 0; i < GRP; ++i) {
              const int e = lane + 32 * (i0 + i), r = e / CH, ch = e % CH;
              const long long tv = __shfl_sync(0xffffffffu, tv_l, r);
              v[i] = make_uint4(0, 0, 0, 0);
              if (tv >= 0) {
                const long long row = tv & ((1LL << 40) - 1);
                if (row < f.pool_tokens)
                  v[i] = ld_stream(pool + (((size_t)f.layer * f.pool_tokens + row) * p.Hkv + hk) * D + ch * 8);
              } else if (yq != p.oob_row) {
                v[i] = ld_stream(cache + (size_t)(yq + r) * D + ch * 8);
              }
            }
#pragma unroll
            for (int i = 0; i < GRP; ++i) {
              const int e = lane + 32 * (i0 + i), r = e / CH, ch = e % CH;
              sts128(stage + q * kPageBytes + page_piece<D>(r, ch), v[i]);
            }
          }
        }
        if (is_k && lane < 8)  // for the rotators: this stage's page sources
          reinterpret_cast<int2 *>(smem + L::kInfo)[st * 8 + lane] = make_int2(src.kind, src.delta);
        fence_proxy_async();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(b_full + st));
      };
      // every key tile of the cluster's range; the value tiles this CTA's
      // first query tile needs
      const int n_mine = is_k ? n : nt[0];
      PageSrc s_next = source(kv_begin);
      int issued = 0;
      for (int j = 0; j < n_mine; ++j) {
        const int st = j % nst;
        const PageSrc s_cur = s_next;
        if (j + 1 < n_mine) s_next = source(kv_begin + j + 1);
        if (j >= nst) {
          const bool ok = mbar_wait(bar(b_empty + st), ((j / nst) - 1) & 1, abort_flag, p.status, detail);
          if (!__all_sync(0xffffffffu, ok)) break;
        }
        issue(st, kv_begin + j, s_cur);
        issued = j + 1;
      }
      if (lane == 0 && *abort_flag) {
        // Let the copies already issued land before the CTA exits.
        for (int j = max(0, issued - nst); j < issued; ++j)
          mbar_wait(bar(b_full + j % nst), (j / nst) & 1, abort_flag, p.status, detail);
      }
    }
  };
  auto role_issuer = [&]() {
    // ===================================================== MMA issuer
    // The whole warp takes part in the named barriers; lane 0 issues.  After
    // an abort both this loop and the relay's run to the end (skipping their
    // waits and MMAs), so every barrier sync has its arrival.
    const bool leader = lane == 0;
    if (leader) mbar_wait(bar(B_Q), 0, abort_flag, p.status, detail);
    __syncwarp();
    tc_fence_after();
    // K(j)'s ring slot is free once every QK reading it has completed -- in
    // rotate-on-load, in both CTAs of the cluster (the peer writes half of it)
    auto release_k = [&](int st) {
      if constexpr (kFused) mma_commit_mc(bar(B_KEMPTY + st), 0x3);
      else mma_commit(bar(B_KEMPTY + st));
    };
    // Matrix descriptors: one base per operand region.  A ring stage, a query
    // tile or a k-step only moves the start address, which sits in the low 14
    // bits as address >> 4; shared addresses stay below 256 KB, so adding
    // (offset >> 4) never carries out of the field.  Built once here, each
    // MMA costs the issuer an add instead of a full descriptor.
    const uint64_t dQ = sdesc_sw128(sbase + L::kQ, 16, 1024);
    const uint64_t dK = sdesc_sw128(sbase + L::kK, 16, kGroupStride);
    const uint64_t dV = sdesc_sw128(sbase + L::kV, kPanelOff, kGroupStride);
    for (int j = 0; j <= n; ++j) {
      bool k_ready = false;
#pragma unroll
      for (int t = 0; t < NQ; ++t) {
        if (t >= ntile) break;
        const uint32_t tS = tbase + t * 128, tO = tbase + 256 + t * 128;
        // O_t += P_t(j-1) V(j-1)
        if (j >= 1 && j - 1 < nt[t]) {
          const int pj = j - 1, pst = pj % NSV;
          named_bar_sync(kNbPv + t, 64);
          tc_fence_after();
          if (leader && !*abort_flag) {
            const uint64_t dv = dV + (uint64_t)((pst * L::kTile) >> 4);
#pragma unroll
            for (int kk = 0; kk < BN / 16; ++kk)  // one page of 16 keys per MMA
              mma_ts(tO, tS + kk * 8, dv + (kk * kPageBytes) / 16, IDESC_PV, (pj > 0 || kk > 0));
            // the last tile that reads V(j-1) releases it (tile 1 reads a prefix of tile 0's range)
            if (t == ntile - 1 || pj >= nt[1]) mma_commit(bar(B_VEMPTY + pst));
          }
        }
        // S_t = Q_t K(j)^T
        if (j < nt[t]) {
          const int st = j % NSK;
          if (!k_ready) {
            named_bar_sync(kNbK, 64);
            tc_fence_after();
            k_ready = true;
          }
          if (leader && !*abort_flag) {
            const uint64_t dk = dK + (uint64_t)((st * L::kTile) >> 4);
            const uint64_t dq = dQ + (uint64_t)((t * L::kQTile) >> 4);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              mma_ss(tS, dq + ((kk >> 2) * (BM * 128) + (kk & 3) * 32) / 16,
                     dk + ((kk >> 2) * kPanelOff + (kk & 3) * 32) / 16, IDESC_QK, kk > 0);
            mma_commit(bar(B_SFULL + t));
            if (t == ntile - 1 || j >= nt[1]) release_k(st);  // last reader of K(j)
          }
        }
      }
      if (kFused && j < n && !k_ready) {
        // A key tile only the cluster peer uses: released once both halves
        // are in this CTA's ring (its rotators are done with it, the peer's
        // copy has landed).  The issuer waits itself rather than through the
        // relay, whose arrivals here would depend on nothing the issuer
        // does and could run a phase ahead of its syncs.
        if (leader) {
          mbar_wait(bar(B_KROT + j % NSK), (j / NSK) & 1, abort_flag, p.status, detail);
          mbar_wait(bar(B_KPEER + j % NSK), (j / NSK) & 1, abort_flag, p.status, detail);
          release_k(j % NSK);
        }
        __syncwarp();
      }
    }
    if (leader) mma_commit(bar(B_OFINAL));
  };
  auto role_relay = [&]() {
    // ===================================================== relay for the issuer
    // Mirrors the issuer's loop: the same conditions, the same order.  Its
    // arrival on a barrier in iteration j + 1 depends on an MMA the issuer
    // issues only after its sync on that barrier in iteration j, so the two
    // never get a phase apart.
    auto wait_k = [&](int j) {  // K(j) complete in this CTA's ring
      const uint32_t par = (j / NSK) & 1;
      if constexpr (kFused) {
        mbar_wait(bar(B_KROT + j % NSK), par, abort_flag, p.status, detail);
        mbar_wait(bar(B_KPEER + j % NSK), par, abort_flag, p.status, detail);
      } else {
        mbar_wait(bar(B_KFULL + j % NSK), par, abort_flag, p.status, detail);
      }
    };
    for (int j = 0; j <= n; ++j) {
      bool k_ready = false, v_ready = false;
#pragma unroll
      for (int t = 0; t < NQ; ++t) {
        if (t >= ntile) break;
        if (j >= 1 && j - 1 < nt[t]) {
          const int pj = j - 1, pst = pj % NSV;
          if (!v_ready) {
            mbar_wait(bar(B_VFULL + pst), (pj / NSV) & 1, abort_flag, p.status, detail);
            v_ready = true;
          }
          mbar_wait(bar(B_PFULL + t), pj & 1, abort_flag, p.status, detail);
          named_bar_arrive(kNbPv + t, 64);
        }
        if (j < nt[t] && !k_ready) {
          wait_k(j);
          named_bar_arrive(kNbK, 64);
          k_ready = true;
        }
      }
    }
  };
  auto role_rotator = [&]() {
    // ===================================================== rotators (rotate-on-load)
    // For every K tile: wait for its pages, rotate each document row by its
    // document's delta exactly as pic_relocate does (cos/sin of the
    // fp64-reduced angle, fp32 rotation, bf16 round to nearest even), then
    // release the tile to the MMA issuer on B_KROT (one arrival per warp).
    // Thread rt takes the 8-pair chunk rt % KC of one row of KC of the
    // tile's pages; its cos/sin are recomputed only when its rows' document
    // changes.
    if constexpr (kFused) {
      // Warp w of the rotators takes page 4 crank + w of each tile (the CTA's
      // half; the cluster peer rotates the other); lane l the 8-pair chunk
      // l % KC of rows l / KC + RG i (i < RPL) of the page.
      constexpr int KC = D / 16, RG = 32 / KC, RPL = 16 / RG;
      const int wr = warp - W_ROT;
      const int my_c = lane % KC, my_rg = lane / KC;
      const PairChunk pc = pair_chunk(my_c, D / 2, rp.style);
      const int2 *info = reinterpret_cast<const int2 *>(smem + L::kInfo);
      // cos/sin of this lane's 8 pairs for document k (64 bytes of the set-up
      // kernel's table, reloaded only when the document changes), kept as the
      // packed fp32 pairs the rotation multiplies by:
      //   half-split:  A[j] = (c_2j, c_2j+1), A[4+j] = (s_2j, s_2j+1),
      //                N[j] = (-s_2j, -s_2j+1)                      (j < 4)
      //   interleaved: A[q] = (c_q, s_q), N[q] = (-s_q, c_q)        (q < 8)
      uint64_t A[8], N[8];
      int cs_doc = -1;
      const bool half_style = rp.style == PIC_ROPE_HALF;
      auto ensure_cs = [&](int k) {
        if (k == cs_doc) return;
        const float4 *src = reinterpret_cast<const float4 *>(
            f.doc_cs + ((size_t)b * f.max_docs + k) * (D / 2) + 8 * my_c);
        float c[8], sn[8];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const float4 v = src[q];
          c[2 * q] = v.x;
          sn[2 * q] = v.y;
          c[2 * q + 1] = v.z;
          sn[2 * q + 1] = v.w;
        }
        if (half_style) {
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            A[j] = f2pack(c[2 * j], c[2 * j + 1]);
            A[4 + j] = f2pack(sn[2 * j], sn[2 * j + 1]);
            N[j] = f2pack(-sn[2 * j], -sn[2 * j + 1]);
          }
        } else {
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            A[q] = f2pack(c[q], sn[q]);
            N[q] = f2pack(-sn[q], c[q]);
          }
        }
        cs_doc = k;
      };
      // Rotates the 8 pairs of one chunk in place, on packed fp32 pairs:
      //   u' = fma(u, c, w * -s),  w' = fma(u, s, w * c)
      // -- per element exactly the operations of the relocation kernel's
      // scalar rotation, so the rounded keys are identical.  The tile loop
      // below is instantiated once per RoPE style, so the warps execute only
      // their style's code (the loop shares the SMSPs' instruction caches
      // with the softmax).
      auto rotate_tiles = [&](auto half_c) {
        constexpr bool kHalf = decltype(half_c)::value;
        auto rot = [&](uint4 &va, uint4 &vb) {
          uint32_t *wa = reinterpret_cast<uint32_t *>(&va), *wb = reinterpret_cast<uint32_t *>(&vb);
          if constexpr (kHalf) {  // va: u of pairs 0..7, vb: w of the same pairs
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint64_t u2 = bf2_to_f2(wa[j]), w2 = bf2_to_f2(wb[j]);
              const uint64_t nu = fma2(u2, A[j], mul2(w2, N[j]));
              const uint64_t nw = fma2(u2, A[4 + j], mul2(w2, A[j]));
              wa[j] = f2_to_bf2(nu);
              wb[j] = f2_to_bf2(nw);
            }
          } else {  // each word one pair (u, w): pairs 0..3 in va, 4..7 in vb
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              uint32_t &wq = q < 4 ? wa[q] : wb[q - 4];
              uint64_t uu, ww;
              f2_split_dup(bf2_to_f2(wq), uu, ww);
              wq = f2_to_bf2(fma2(uu, A[q], mul2(ww, N[q])));
            }
          }
        };
        for (int j = 0; j < n; ++j) {
          const int st = j % NSK;
          const bool ok = __all_sync(0xffffffffu, mbar_wait(bar(B_KFULL + st), (j / NSK) & 1,
                                                             abort_flag, p.status, detail));
          const uint32_t stage = sbase + L::kK + st * L::kTile;
          const int q = 4 * (int)crank + wr;  // this warp's page: one of the CTA's half
          const int2 pi = info[st * 8 + q];
          if (ok && pi.x != 0) {
            const uint32_t pbase = stage + q * kPageBytes;
            // a row at a time (a rolled loop keeps the rotators' code small in
            // the instruction caches they share with the softmax): a page of
            // one document rotates every row by that document's delta, a page
            // across a boundary each row by its own document's, inline rows
            // stay as they are
            const int16_t *rd = reinterpret_cast<const int16_t *>(smem + L::kRowDoc) + (st * 8 + q) * 16;
#pragma unroll 1
            for (int i = 0; i < RPL; ++i) {
              const int r = my_rg + RG * i;
              const int kd = pi.x == 1 ? pi.y : rd[r];
              if (kd < 0) continue;
              ensure_cs(kd);
              const uint32_t a0 = pbase + page_piece<D>(r, pc.off_a / 8);
              const uint32_t a1 = pbase + page_piece<D>(r, pc.off_b / 8);
              uint4 va = lds128(a0), vb = lds128(a1);
              rot(va, vb);
              sts128(a0, va);
              sts128(a1, vb);
            }
          }
          fence_proxy_async();
          __syncwarp();
          // the page rotated: a bulk copy into the same slot of the cluster
          // peer, whose K(j) is complete when these four pages and its own
          // half are
          if (lane == 0) {
            if (!*abort_flag) {
              const uint32_t page = stage + q * kPageBytes;
              bulk_copy_to_peer(map_to_rank(page, cpeer), page, kPageBytes,
                                map_to_rank(bar(B_KPEER + st), cpeer));
            }
            mbar_arrive(bar(B_KROT + st));
          }
        }
      };
      if (half_style) rotate_tiles(std::true_type{});
      else rotate_tiles(std::false_type{});
    }
  };
  auto role_softmax = [&]() {
    // ===================================================== softmax warpgroups
    static_assert(NQ == 2, "softmax warpgroup selection assumes two query tiles");
    const int t = (warp - W_SM) >> 2;  // query tile of this warpgroup
    const int wq = warp & 3;        // TMEM lane quarter
    const int row = wq * 32 + lane;
    // constant-index selects keep the per-tile values in registers
    const int my_r0 = t == 0 ? r0[0] : r0[1];
    const int my_kmin = t == 0 ? kmin[0] : kmin[1];
    const int my_n = t < ntile ? (t == 0 ? nt[0] : nt[1]) : 0;
    const size_t my_part0 = part_row0(t);
    const int rg = my_r0 + row;
    const bool valid = t < ntile && rg >= 0 && rg < rows;
    const int tok = valid ? rg / p.G : 0, g = valid ? rg % p.G : 0;
    const int pos = valid ? ipos[tok] : -1;
    const uint32_t tl = tbase + ((uint32_t)(wq * 32) << 16);
    const uint32_t tS = tl + t * 128, tO = tl + 256 + t * 128;
    float m_used = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < my_n; ++j) {
      const int key0 = (kv_begin + j) * BN;
      if (!__all_sync(0xffffffffu, mbar_wait(bar(B_SFULL + t), j & 1, abort_flag, p.status, detail))) {
        ok = false;
        break;
      }
      tc_fence_after();
      float s[BN];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c) tmem_ld32(tS + c * 32, reinterpret_cast<uint32_t *>(s + c * 32));
      tmem_wait_ld();
      if (key0 + BN - 1 > my_kmin) {  // some key of the tile lies beyond some row
#pragma unroll
        for (int c = 0; c < BN; ++c)
          if (key0 + c > pos) s[c] = -INFINITY;
      }
      // Exponents against the running maximum m_used.  From the second tile
      // on, a warp whose rows all have one skips the row maximum and
      // exponentiates against m_used directly; the tile's row sum then bounds
      // every exponential, and if some row's sum reaches 2^64 (its scores grew
      // by more than 64 in the log2 domain) the tile is redone the first way:
      // row maximum, rescale when it grew by more than 2^8, exponentials again.
      // P (bf16) up to 2^64 and the fp32 sums of a few thousand of them stay
      // far inside the range of both.
      float alpha = 1.f;
      bool resc = false;
      bool need_max = !__all_sync(0xffffffffu, j > 0 && m_used != -INFINITY);
      float l0, l1;
#pragma unroll 1
      for (int pass = 0; pass < 2; ++pass) {
        if (need_max) {
          // row max: 4 independent chains of 3-input max
          float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
          for (int c = 0; c < BN; c += 8)
#pragma unroll
            for (int i = 0; i < 4; ++i) mx[i] = max3f(mx[i], s[c + 2 * i], s[c + 2 * i + 1]);
          const float m_new = fmaxf(m_used, max3f(mx[0], mx[1], fmaxf(mx[2], mx[3])) * p.scale_log2);
          resc = m_new > m_used + 8.f;
          if (resc) {
            alpha = ex2(m_used - m_new);
            m_used = m_new;
          }
        }
        const float mref = (m_used == -INFINITY) ? 0.f : m_used;
        // P = exp2(s * scale - m) as bf16, written over S in 16-column chunks
        // as soon as each 32-key chunk is done (S was read completely above,
        // so the overlap is harmless and the packed values never pile up in
        // registers).  Scaling and the row sum run on packed fp32 pairs (half
        // the issue slots; the softmax is bound by instruction issue, not by
        // MUFU).
        const uint64_t sc2 = f2pack(p.scale_log2, p.scale_log2), nm2 = f2pack(-mref, -mref);
        uint64_t acc[4] = {0, 0, 0, 0};
#pragma unroll
        for (int c0 = 0; c0 < BN; c0 += 32) {
          uint32_t pk[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const uint64_t e = exp2_mufu2(fma2(f2pack(s[c0 + 2 * q], s[c0 + 2 * q + 1]), sc2, nm2));
            acc[q & 3] = add2(acc[q & 3], e);
            float e0, e1;
            f2unpack(e, e0, e1);
            pk[q] = pack2(e0, e1);
          }
          tmem_st16(tS + c0 / 2, pk);
        }
        acc[0] = add2(add2(acc[0], acc[1]), add2(acc[2], acc[3]));
        f2unpack(acc[0], l0, l1);
        if (need_max || !__any_sync(0xffffffffu, !(l0 + l1 < 0x1p64f))) break;
        need_max = true;
      }
      l = fmaf(l, alpha, l0 + l1);
      // O correction: PV_t(j-1) has completed (it precedes QK_t(j) in the MMA order)
      if (j > 0 && __any_sync(0xffffffffu, resc)) {
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(tO + c * 32, reinterpret_cast<uint32_t *>(o));
          tmem_wait_ld();
#pragma unroll
          for (int q = 0; q < 32; ++q) o[q] *= alpha;
          tmem_st32(tO + c * 32, reinterpret_cast<uint32_t *>(o));
        }
      }
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_PFULL + t));  // one arrival per warp
    }
    // ---- epilogue
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar(B_OFINAL), 0, abort_flag, p.status, detail));
    tc_fence_after();
    if (t < ntile && my_n == 0) {  // this tile needs none of the split's keys
      if (ok && p.num_splits > 1) {
        p.part_ml[(my_part0 + row) * 2] = -INFINITY;
        p.part_ml[(my_part0 + row) * 2 + 1] = 0.f;
      }
    } else if (t < ntile) {
      // Every MMA and TMA copy is finished, so the whole shared memory is free:
      // each thread stages its finished row (padded rows keep the bank
      // accesses at 4 wavefronts per 512 B), the warpgroup syncs on its own
      // named barrier, and warps copy whole rows out with coalesced stores.
      const bool single = p.num_splits == 1;
      constexpr int kRowOut = D * 2 + 16;  // a row of bf16 outputs or fp16 partials, padded
      uint8_t *stage = smem + (size_t)t * BM * kRowOut;
      if (ok) {
        float o[D];
#pragma unroll
        for (int c = 0; c < D / 32; ++c) tmem_ld32(tO + c * 32, reinterpret_cast<uint32_t *>(o + c * 32));
        tmem_wait_ld();
        if (single) {
          const float inv = l > 0.f ? 1.f / l : 0.f;
          uint4 *dst = reinterpret_cast<uint4 *>(stage + row * kRowOut);
#pragma unroll
          for (int q = 0; q < D; ++q) o[q] *= inv;
#pragma unroll
          for (int q = 0; q < D / 8; ++q) dst[q] = pack8(o + q * 8);
          if (valid && p.lse)
            p.lse[((size_t)b * p.max_inline + tok) * p.Hq + hk * p.G + g] =
                l > 0.f ? (m_used + __log2f(l)) * 0.69314718055994531f : -INFINITY;
        } else {
          // a split's partial row: O / l in fp16 (|O / l| is at most the
          // largest |v|), with m and l beside it for the merge's weights
          const float inv = l > 0.f ? 1.f / l : 0.f;
          uint4 *dst = reinterpret_cast<uint4 *>(stage + row * kRowOut);
#pragma unroll
          for (int q = 0; q < D; ++q) o[q] *= inv;
#pragma unroll
          for (int q = 0; q < D / 8; ++q) dst[q] = pack8_h(o + q * 8);
          p.part_ml[(my_part0 + row) * 2] = (l > 0.f) ? m_used : -INFINITY;
          p.part_ml[(my_part0 + row) * 2 + 1] = l;
        }
      }
      asm volatile("bar.sync %0, 128;" ::"r"(1 + t) : "memory");
      if (ok) {
        const int rlo = max(0, -my_r0);  // the tile's rows from rlo on exist
        if (single) {
          // 16 lanes per 256-byte row (D = 128) or 8 per 128-byte row (D = 64)
          constexpr int LPR = D / 8, RPI = 32 / LPR;
          for (int r = wq * RPI + lane / LPR; r < BM; r += 4 * RPI) {
            if (r < rlo) continue;
            const int rg2 = my_r0 + r, tk = rg2 / p.G, gg = rg2 % p.G;
            const uint4 v = *reinterpret_cast<const uint4 *>(stage + r * kRowOut + (lane % LPR) * 16);
            st_global16(p.out + (((size_t)b * p.max_inline + tk) * p.Hq + hk * p.G + gg) * D +
                            (lane % LPR) * 8, v);
          }
        } else {
          // the partial rows are contiguous in the partial buffer
          constexpr int LPR = D / 8, RPI = 32 / LPR;
          for (int r = wq * RPI + lane / LPR; r < BM; r += 4 * RPI) {
            if (r < rlo) continue;
            const uint4 v = *reinterpret_cast<const uint4 *>(stage + r * kRowOut + (lane % LPR) * 16);
            *reinterpret_cast<uint4 *>(p.part_o + (my_part0 + r) * D + (lane % LPR) * 8) = v;
          }
        }
      }
    }
  };
  if constexpr (kFused) {
    if constexpr (kGroup == 0) {
      if (warp == 0 || warp == W_V) role_producer();
      else if (warp == 1) role_issuer();
      else role_relay();
    } else if constexpr (kGroup == 1) {
      role_rotator();
    } else {
      role_softmax();
    }
  } else {
    if (warp == 0 || warp == W_V) role_producer();
    else if (warp == 1) role_issuer();
    else if (warp == W_RELAY) role_relay();
    else role_softmax();
  }
  // Release the dependent launch (the split merge, or the next layer's
  // append) only now: released at the start, it made the pass slower.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  tc_fence_before();
  __syncthreads();
  if constexpr (kFused) {
    // Leave only when the cluster peer is done too: its last copies into this
    // CTA's ring have landed (the relay waited for them) and it no longer
    // reads the copies this CTA sent.  The wait is bounded even after an abort.
    if (threadIdx.x == 0) {
      mbar_arrive_remote(map_to_rank(bar(B_EXIT), cpeer));
      volatile int keep_waiting = 0;
      mbar_wait(bar(B_EXIT), 0, &keep_waiting, p.status, detail);
    }
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    if (*abort_flag && lane == 0) {
      // make sure no MMA is still running on the TMEM we are about to free
      mbar_wait(bar(B_OFINAL), 0, abort_flag, p.status, detail);
    }
    __syncwarp();
    tmem_dealloc(tbase, kTmemCols);
  }
}

template <int D, bool kFused>
__global__ void __launch_bounds__(threads_of<kFused>(), 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_kp,
                const __grid_constant__ CUtensorMap tm_vp, Params p, FusedArgs f, RopeParams rp) {
  if constexpr (kFused) {
    // Registers move from the control and rotator warpgroups to the softmax
    // ones: each warpgroup runs one setmaxnreg, first thing, and then its
    // own copy of the body.
    const int wg = threadIdx.x >> 7;
    if (wg == 0) {
      asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegCtl));
      attn_body<D, true, 0>(tm_q, tm_k, tm_v, tm_kp, tm_vp, p, f, rp);
    } else if (wg == 3) {
      asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegRot));
      attn_body<D, true, 1>(tm_q, tm_k, tm_v, tm_kp, tm_vp, p, f, rp);
    } else {
      asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegSoftmax));
      attn_body<D, true, 2>(tm_q, tm_k, tm_v, tm_kp, tm_vp, p, f, rp);
    }
  } else {
    attn_body<D, false, -1>(tm_q, tm_k, tm_v, tm_kp, tm_vp, p, f, rp);
  }
}


// Merge the split partials (O / l in fp16, m in log2 units, l) of every
// query row by log-sum-exp -- o = sum_s w_s (O_s / l_s) / sum_s w_s with
// w_s = 2^(m_s - M) l_s -- lanes over the d columns.  A warp takes R rows of
// one query tile and issues the (m, l) pairs and the O rows of U splits for
// all R rows before using any of them (R * U = 8 loads in flight per lane),
// so a row costs one L2/DRAM round trip for up to U splits;
// U is the smallest of 2, 4, 8 that covers the splits (more are merged in
// further rounds).  An empty split's weight is zero and its data, never
// written, is discarded by a select.  Launched as a programmatic dependent of
// the attention kernel: the CTAs may be placed while attention drains and
// wait for it here.
template <int D, int U, int R>
__global__ void __launch_bounds__(256) combine_kernel(Params p) {
  constexpr int CPL = D / 32;
  static_assert(BM % R == 0, "a warp's rows stay inside one query tile");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long g0 = ((long long)blockIdx.x * (blockDim.x >> 5) + warp) * R;
  const long long per_b = (long long)p.Hkv * p.m_tiles * BM;
  const int b = (int)(g0 / per_b);
  if (b >= p.batch) return;
  const long long rem = g0 % per_b;
  const int hk = (int)(rem / ((long long)p.m_tiles * BM));
  const int mt = (int)((rem / BM) % p.m_tiles), row0 = (int)(rem % BM);
  const int tin = min(max(p.inline_len[b], 0), p.max_inline);
  // the warp's rows are rg0 .. rg0 + R - 1 of the request (tiles counted
  // from its last row); those below row 0 are padding
  const int rg0 = tin * p.G - (mt + 1) * BM + row0;
  if (rg0 + R <= 0) return;
  const int S = p.num_splits;
  const size_t base = (((size_t)b * p.Hkv + hk) * p.m_tiles + mt) * S;
  float ms[R], ls[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    ms[r] = -INFINITY, ls[r] = 0.f;
    if (lane < S) {
      const float2 ml =
          *reinterpret_cast<const float2 *>(p.part_ml + ((base + lane) * BM + row0 + r) * 2);
      ms[r] = ml.x, ls[r] = ml.y;
    }
  }
  float acc[R][CPL], M[R], w[R], Lsum[R];
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int q = 0; q < CPL; ++q) acc[r][q] = 0.f;
  for (int s0 = 0; s0 < S; s0 += U) {
    float v[R][U][CPL];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int sp = min(s0 + u, S - 1);  // past the end: a harmless reload, weight 0 below
        const __half *src = p.part_o + ((base + sp) * BM + row0 + r) * D + lane * CPL;
        if constexpr (CPL == 4) {
          const uint2 x = *reinterpret_cast<const uint2 *>(src);
          const float2 a = __half22float2(*reinterpret_cast<const __half2 *>(&x.x));
          const float2 c = __half22float2(*reinterpret_cast<const __half2 *>(&x.y));
          v[r][u][0] = a.x, v[r][u][1] = a.y, v[r][u][2] = c.x, v[r][u][3] = c.y;
        } else {
          static_assert(CPL == 2, "d = 64 or 128");
          const float2 a = __half22float2(*reinterpret_cast<const __half2 *>(src));
          v[r][u][0] = a.x, v[r][u][1] = a.y;
        }
      }
    if (s0 == 0) {
#pragma unroll
      for (int r = 0; r < R; ++r) {
        M[r] = ms[r];
#pragma unroll
        for (int o = 16; o; o >>= 1) M[r] = fmaxf(M[r], __shfl_xor_sync(0xffffffffu, M[r], o));
        // weight of split `lane` for the normalised partial: exp2(m_s - M) l_s
        w[r] = (ms[r] == -INFINITY) ? 0.f : ex2(ms[r] - M[r]) * ls[r];
        Lsum[r] = w[r];
#pragma unroll
        for (int o = 16; o; o >>= 1) Lsum[r] += __shfl_xor_sync(0xffffffffu, Lsum[r], o);
      }
    }
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const float ws = __shfl_sync(0xffffffffu, w[r], (s0 + u) & 31);
        const bool use = s0 + u < S && ws != 0.f;
#pragma unroll
        for (int q = 0; q < CPL; ++q)
          acc[r][q] = fmaf(use ? ws : 0.f, use ? v[r][u][q] : 0.f, acc[r][q]);
      }
  }
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int rg = rg0 + r;
    if (rg < 0) continue;
    const float inv = Lsum[r] > 0.f ? 1.f / Lsum[r] : 0.f;
    const int tok = rg / p.G, g = rg % p.G;
    __nv_bfloat16 *dst =
        p.out + (((size_t)b * p.max_inline + tok) * p.Hq + hk * p.G + g) * D + lane * CPL;
#pragma unroll
    for (int q = 0; q < CPL; q += 2)
      *reinterpret_cast<uint32_t *>(dst + q) = pack2(acc[r][q] * inv, acc[r][q + 1] * inv);
    if (p.lse && lane == 0)
      p.lse[((size_t)b * p.max_inline + tok) * p.Hq + hk * p.G + g] =
          Lsum[r] > 0.f ? (M[r] + __log2f(Lsum[r])) * 0.69314718055994531f : -INFINITY;
  }
}

// RoPE the inline keys/queries at their logical positions; keys and values go
// to their cache slots, queries to the GQA-packed workspace.
struct AppendArgs {
  int Hq, Hkv, G, max_inline, max_ctx, R_pad, layer, max_pages;
  long long num_pages;
  const __nv_bfloat16 *q, *k, *v;
  const int32_t *inline_pos, *inline_len;
  const int64_t *slots;          // slot map, or NULL: slots from the block table
  const int32_t *block_table;
  __nv_bfloat16 *k_cache, *v_cache, *qpack;  // cache pointers already at the layer
  int32_t *status;
};

template <int D>
__global__ void __launch_bounds__(256) append_kernel(AppendArgs a, RopeParams rp) {
  constexpr int HALF = D / 2, KC = D / 16, VC = D / 8;
  pdl_entry();
  const int t = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int tin = min(max(a.inline_len[b], 0), a.max_inline);
  __shared__ float2 cs[HALF];
  if (t >= tin) {  // zero the packed query rows of this token slot
    for (int e = tid; e < a.Hkv * a.G * VC; e += blockDim.x) {
      const int hk = e / (a.G * VC), r = e % (a.G * VC), g = r / VC, c = r % VC;
      const int row = t * a.G + g;
      if (row < a.R_pad)
        st_global16(a.qpack + (((size_t)b * a.Hkv + hk) * a.R_pad + row) * D + c * 8,
                    make_uint4(0, 0, 0, 0));
    }
    return;
  }
  const size_t tok = (size_t)b * a.max_inline + t;
  const int nQ = a.Hq * KC, nK = a.Hkv * KC, nV = a.Hkv * VC;
  // First round of loads goes out before the position is even known.
  uint4 qa = make_uint4(0, 0, 0, 0), qb = qa, ka = qa, kb = qa, vv = qa;
  const PairChunk pq = pair_chunk(tid % KC, HALF, rp.style);
  if (tid < nQ) {
    const __nv_bfloat16 *src = a.q + (tok * a.Hq + tid / KC) * D;
    qa = ld_stream(src + pq.off_a);
    qb = ld_stream(src + pq.off_b);
  }
  if (tid < nK) {
    const __nv_bfloat16 *src = a.k + (tok * a.Hkv + tid / KC) * D;
    ka = ld_stream(src + pq.off_a);
    kb = ld_stream(src + pq.off_b);
  }
  if (tid < nV) vv = ld_stream(a.v + (tok * a.Hkv + tid / VC) * D + (tid % VC) * 8);

  const int pos = a.inline_pos[tok];
  const bool pos_ok = pos >= 0 && pos < a.max_ctx;
  long long slot = -1;
  if (pos_ok) {
    if (a.slots) {
      slot = a.slots[(size_t)b * a.max_ctx + pos];
    } else if ((pos >> 4) < a.max_pages) {
      slot = (long long)a.block_table[(size_t)b * a.max_pages + (pos >> 4)] * 16 + (pos & 15);
    } else {
      if (tid == 0) dev_fail(a.status, PIC_DEV_BLOCK_TABLE_SHORT, b);
      slot = -2;
    }
  }
  if (!pos_ok) {
    if (tid == 0) dev_fail(a.status, PIC_DEV_BAD_POSITION, b);
  } else if (slot == -2) {
    slot = -1;
  } else if (slot < 0 || slot >= a.num_pages * 16) {
    if (tid == 0) dev_fail(a.status, PIC_DEV_BAD_PAGE, b);
    slot = -1;
  }
  for (int i = tid; i < HALF; i += blockDim.x)
    cs[i] = rope_cos_sin(pos_ok ? pos : 0, rope_theta(rp, a.layer, i));
  __syncthreads();
  const long long page = slot >> 4, r = slot & 15;

  auto rot_store = [&](uint4 xa, uint4 xb, int c, __nv_bfloat16 *dst) {
    float x[8], y[8], u[8], w[8];
    unpack8(xa, x);
    unpack8(xb, y);
    if (rp.style == PIC_ROPE_HALF) {
#pragma unroll
      for (int i = 0; i < 8; ++i) { u[i] = x[i]; w[i] = y[i]; }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        u[i] = x[2 * i]; w[i] = x[2 * i + 1];
        u[4 + i] = y[2 * i]; w[4 + i] = y[2 * i + 1];
      }
    }
    rotate8(u, w, cs + 8 * c);
    if (rp.style == PIC_ROPE_HALF) {
#pragma unroll
      for (int i = 0; i < 8; ++i) { x[i] = u[i]; y[i] = w[i]; }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        x[2 * i] = u[i]; x[2 * i + 1] = w[i];
        y[2 * i] = u[4 + i]; y[2 * i + 1] = w[4 + i];
      }
    }
    const PairChunk pc = pair_chunk(c, HALF, rp.style);
    st_global16(dst + pc.off_a, pack8(x));
    st_global16(dst + pc.off_b, pack8(y));
  };
  auto q_dst = [&](int h) {
    const int hk = h / a.G, g = h % a.G;
    return a.qpack + (((size_t)b * a.Hkv + hk) * a.R_pad + (size_t)t * a.G + g) * D;
  };
  if (tid < nQ) rot_store(qa, qb, tid % KC, q_dst(tid / KC));
  if (slot >= 0) {
    if (tid < nK)
      rot_store(ka, kb, tid % KC, a.k_cache + ((page * a.Hkv + tid / KC) * 16 + r) * D);
    if (tid < nV)
      st_global16(a.v_cache + ((page * a.Hkv + tid / VC) * 16 + r) * D + (tid % VC) * 8, vv);
  }
  // remaining rounds (more than 256 tasks of a kind: very wide models)
  for (int e = tid + blockDim.x; e < nQ; e += blockDim.x) {
    const int h = e / KC, c = e % KC;
    rotate_chunk(a.q + (tok * a.Hq + h) * D, q_dst(h), c, HALF, rp.style, cs + 8 * c, true);
  }
  if (slot >= 0) {
    for (int e = tid + blockDim.x; e < nK; e += blockDim.x) {
      const int h = e / KC, c = e % KC;
      rotate_chunk(a.k + (tok * a.Hkv + h) * D, a.k_cache + ((page * a.Hkv + h) * 16 + r) * D, c,
                   HALF, rp.style, cs + 8 * c, true);
    }
    for (int e = tid + blockDim.x; e < nV; e += blockDim.x) {
      const int h = e / VC, c = e % VC;
      st_global16(a.v_cache + ((page * a.Hkv + h) * 16 + r) * D + c * 8,
                  ld_stream(a.v + (tok * a.Hkv + h) * D + c * 8));
    }
  }
}

struct Plan {
  int G, m_tiles, R_pad, splits, n_pidx;
  size_t q_bytes, po_bytes, pml_bytes, total;
};

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

inline Plan plan(const pic_geom_t *g, int batch, int max_inline, int max_ctx, int num_splits) {
  Plan pl;
  pl.G = g->num_q_heads / g->num_kv_heads;
  pl.m_tiles = (int)(((long long)max_inline * pl.G + BM - 1) / BM);
  pl.R_pad = pl.m_tiles * BM;
  const int kv_tiles = (max_ctx + BN - 1) / BN;
  if (num_splits <= 0) {
    // Wave-aware choice: minimise waves * (tiles per split + fixed cost).
    const long long ctas = (long long)batch * g->num_kv_heads * ((pl.m_tiles + NQ - 1) / NQ);
    double best_cost = 1e300;
    num_splits = 1;
    for (int s = 1; s <= std::min(kMaxSplits, std::max(1, kv_tiles)); ++s) {
      const long long waves = (ctas * s + 151) / 152;
      const double cost = (double)waves * ((kv_tiles + s - 1) / s + 2) + (s > 1 ? 2.0 : 0.0);
      if (cost < best_cost - 1e-9) {
        best_cost = cost;
        num_splits = s;
      }
    }
  }
  pl.splits = num_splits;
  pl.q_bytes = align256((size_t)batch * g->num_kv_heads * pl.R_pad * g->head_dim * 2);
  if (pl.splits > 1) {
    const size_t rows = (size_t)batch * g->num_kv_heads * pl.m_tiles * pl.splits * BM;
    pl.po_bytes = align256(rows * g->head_dim * 2);
    pl.pml_bytes = align256(rows * 2 * 4);
  } else {
    pl.po_bytes = pl.pml_bytes = 0;
  }
  pl.n_pidx = (max_ctx + 15) / 16;
  pl.total = pl.q_bytes + pl.po_bytes + pl.pml_bytes;
  return pl;
}

// Rotate-on-load's extra workspace, after the plan's: the source of every
// page of positions < max_ctx, then the cos/sin of every listed document.
inline size_t fused_page_bytes(const Plan &pl, int batch) {
  return align256((size_t)batch * pl.n_pidx * sizeof(PageSrcEntry));
}
inline size_t fused_cs_bytes(const pic_geom_t *g, int batch, int max_docs) {
  return align256((size_t)batch * std::max(max_docs, 1) * (g->head_dim / 2) * sizeof(float2));
}

}  // namespace prefill
}  // namespace pic

namespace pic {
namespace prefill {
// The merge kernel as a programmatic dependent launch of the attention
// kernel before it on the stream (it waits with griddepcontrol.wait).
template <int D>
static cudaError_t launch_combine(long long rows, const Params &pp, cudaStream_t stream) {
  const int S = pp.num_splits;
  const int U = S <= 2 ? 2 : (S <= 4 ? 4 : 8), R = 8 / U;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((rows + 8 * R - 1) / (8 * R)));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (U == 2) return cudaLaunchKernelEx(&cfg, combine_kernel<D, 2, 4>, pp);
  if (U == 4) return cudaLaunchKernelEx(&cfg, combine_kernel<D, 4, 2>, pp);
  return cudaLaunchKernelEx(&cfg, combine_kernel<D, 8, 1>, pp);
}
}  // namespace prefill
}  // namespace pic

extern "C" size_t pic_prefill_fused_workspace_size(const pic_geom_t *geom, int32_t batch,
                                                   int32_t max_inline, int32_t max_ctx,
                                                   int32_t max_docs, int32_t num_splits) {
  if (!geom || batch <= 0 || max_inline <= 0 || max_ctx <= 0 || max_docs < 0 ||
      geom->num_kv_heads <= 0 || geom->num_q_heads % geom->num_kv_heads)
    return 0;
  const pic::prefill::Plan pl = pic::prefill::plan(geom, batch, max_inline, max_ctx, num_splits);
  return pl.total + pic::prefill::fused_page_bytes(pl, batch) +
         pic::prefill::fused_cs_bytes(geom, batch, max_docs);
}

extern "C" size_t pic_prefill_workspace_size(const pic_geom_t *geom, int32_t batch,
                                             int32_t max_inline, int32_t max_ctx,
                                             int32_t num_splits) {
  if (!geom || batch <= 0 || max_inline <= 0 || max_ctx <= 0 || geom->num_kv_heads <= 0 ||
      geom->num_q_heads % geom->num_kv_heads)
    return 0;
  return pic::prefill::plan(geom, batch, max_inline, max_ctx, num_splits).total;
}

namespace pic {
namespace prefill {

// Checks shared by pic_append_inline and pic_attend_prefill.
static pic_status_t check_common(const char *who, const pic_geom_t *geom, int32_t layer,
                                 int32_t batch, int32_t max_inline, int32_t max_ctx,
                                 int64_t num_pages, int32_t num_splits, void *workspace,
                                 size_t workspace_bytes, RopeParams *rp, Plan *pl) {
  pic_status_t st = make_rope(geom, rp);
  if (st != PIC_OK) return st;
  if (layer < 0 || layer >= geom->num_layers)
    return fail(PIC_ERR_INVALID_ARG, "%s: layer %d outside [0, %d)", who, layer, geom->num_layers);
  if (batch <= 0 || max_inline <= 0 || max_ctx <= 0 || num_pages <= 0)
    return fail(PIC_ERR_INVALID_ARG, "%s: sizes must be positive", who);
  if (num_splits < 0 || num_splits > kMaxSplits)
    return fail(PIC_ERR_INVALID_ARG, "%s: num_splits %d outside [0, %d]", who, num_splits,
                kMaxSplits);
  const long long rows_total = (long long)geom->num_layers * num_pages * geom->num_kv_heads * 16;
  if (rows_total + 16 >= (long long)INT32_MAX)
    return fail(PIC_ERR_UNSUPPORTED, "%s: cache has more than 2^31 rows", who);
  *pl = plan(geom, batch, max_inline, max_ctx, num_splits);
  if ((long long)batch * geom->num_kv_heads * pl->R_pad >= (long long)INT32_MAX ||
      pl->m_tiles * pl->splits > 65535 || geom->num_kv_heads > 65535 || batch > 65535)
    return fail(PIC_ERR_UNSUPPORTED, "%s: problem too large for one launch", who);
  if (!workspace || workspace_bytes < pl->total || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return fail(PIC_ERR_WORKSPACE, "%s: workspace needs %zu bytes, 256-aligned", who, pl->total);
  return PIC_OK;
}

}  // namespace prefill
}  // namespace pic

extern "C" int32_t pic_prefill_num_splits(const pic_geom_t *geom, int32_t batch,
                                          int32_t max_inline, int32_t max_ctx,
                                          int32_t num_splits) {
  if (!geom || batch <= 0 || max_inline <= 0 || max_ctx <= 0 || geom->num_kv_heads <= 0 ||
      geom->num_q_heads % geom->num_kv_heads || num_splits < 0 ||
      num_splits > pic::prefill::kMaxSplits)
    return 0;
  return pic::prefill::plan(geom, batch, max_inline, max_ctx, num_splits).splits;
}

// Key-split count for the requests' actual inline positions: for every
// candidate count, the attention grid's CTAs in launch order (one per query
// pair, key split, kv head and request, a pair's tiles counted from the
// request's last packed row as the kernel does) are dealt greedily to the
// SMs, each costing its key tiles plus a fixed per-CTA cost, and the count
// with the least makespan (plus a merge cost when split) wins; a grid that
// fits in one wave with the library's count is not split further.
extern "C" int32_t pic_prefill_plan_splits(const pic_geom_t *geom, int32_t batch,
                                           int32_t max_inline, int32_t max_ctx,
                                           const int32_t *inline_len, const int32_t *inline_pos) {
  using namespace pic::prefill;
  if (!inline_len || !inline_pos) return 0;
  const int32_t fallback = pic_prefill_num_splits(geom, batch, max_inline, max_ctx, 0);
  if (fallback <= 0) return 0;
  const int G = geom->num_q_heads / geom->num_kv_heads, Hkv = geom->num_kv_heads;
  const int m_tiles = (int)(((long long)max_inline * G + BM - 1) / BM), npairs = (m_tiles + NQ - 1) / NQ;
  const int kv_tiles = (max_ctx + BN - 1) / BN;
  // key tiles of each (request, pair): 0 for a pair without rows
  std::vector<int> pair_tiles((size_t)batch * npairs, 0);
  for (int b = 0; b < batch; ++b) {
    const int tin = std::min(std::max(inline_len[b], 0), max_inline);
    const int rows = tin * G;
    for (int pr = 0; pr < npairs; ++pr) {
      const int r0 = rows - (pr * NQ + 1) * BM;
      if (pr * NQ < m_tiles && r0 + BM > 0) {
        const int kmax = inline_pos[(size_t)b * max_inline + (r0 + BM - 1) / G];
        pair_tiles[(size_t)b * npairs + pr] = kmax >= 0 ? std::min(kmax / BN + 1, kv_tiles) : 0;
      }
    }
  }
  constexpr double kCtaFixed = 2.0, kCtaEmpty = 0.3, kMerge = 1.0;  // in key-tile times
  constexpr int kSms = 152;
  double best = 1e300;
  int best_s = fallback;
  std::vector<double> sm(kSms);
  // A grid the library's count already fits in one wave is latency-bound:
  // more splits there only add merge traffic the estimate leaves out.
  int max_s = std::min(kMaxSplits, std::max(1, kv_tiles));
  if ((long long)batch * Hkv * npairs * fallback <= kSms) max_s = std::min(max_s, fallback);
  for (int sp = 1; sp <= max_s; ++sp) {
    std::fill(sm.begin(), sm.end(), 0.0);
    std::make_heap(sm.begin(), sm.end(), std::greater<double>());
    for (int b = 0; b < batch; ++b)
      for (int hk = 0; hk < Hkv; ++hk)
        for (int x = 0; x < npairs * sp; ++x) {
          const int pr = x % npairs, split = x / npairs;
          const int na = pair_tiles[(size_t)b * npairs + pr];
          const int per = (na + sp - 1) / sp;
          const int n = std::max(0, std::min(per, na - split * per));
          std::pop_heap(sm.begin(), sm.end(), std::greater<double>());
          sm.back() += n > 0 ? n + kCtaFixed : kCtaEmpty;
          std::push_heap(sm.begin(), sm.end(), std::greater<double>());
        }
    const double cost = *std::max_element(sm.begin(), sm.end()) + (sp > 1 ? kMerge : 0.0);
    if (cost < best - 1e-9) {
      best = cost;
      best_s = sp;
    }
  }
  return best_s;
}

namespace pic {
namespace prefill {

// One layer's inline append (append_kernel) into the packed-query part of
// the workspace; slots from slot_mapping, or from the block table when it is
// NULL.  Shared by pic_append_inline and the prefill calls that are given
// the projections.
static pic_status_t launch_append(const char *who, const pic_geom_t *geom, const RopeParams &rp,
                                  const Plan &pl, int32_t layer, int32_t batch, int32_t max_inline,
                                  const void *q, const void *k_new, const void *v_new,
                                  const int32_t *inline_pos, const int32_t *inline_len,
                                  const int64_t *slot_mapping, const int32_t *block_table,
                                  int32_t max_pages, int32_t max_ctx, int64_t num_pages,
                                  void *k_cache, void *v_cache, void *workspace,
                                  pic_stream_t stream) {
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k_new) |
       reinterpret_cast<uintptr_t>(v_new) | reinterpret_cast<uintptr_t>(k_cache) |
       reinterpret_cast<uintptr_t>(v_cache)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "%s: bf16 tensors must be 16-byte aligned", who);
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "%s: no device status word", who);
  const int D = geom->head_dim, Hkv = geom->num_kv_heads;
  const size_t layer_elems = (size_t)num_pages * Hkv * 16 * D;
  AppendArgs aa;
  aa.Hq = geom->num_q_heads;
  aa.Hkv = Hkv;
  aa.G = pl.G;
  aa.max_inline = max_inline;
  aa.max_ctx = max_ctx;
  aa.R_pad = pl.R_pad;
  aa.layer = layer;
  aa.max_pages = max_pages;
  aa.num_pages = num_pages;
  aa.q = static_cast<const __nv_bfloat16 *>(q);
  aa.k = static_cast<const __nv_bfloat16 *>(k_new);
  aa.v = static_cast<const __nv_bfloat16 *>(v_new);
  aa.inline_pos = inline_pos;
  aa.inline_len = inline_len;
  aa.slots = slot_mapping;
  aa.block_table = block_table;
  aa.k_cache = static_cast<__nv_bfloat16 *>(k_cache) + (size_t)layer * layer_elems;
  aa.v_cache = static_cast<__nv_bfloat16 *>(v_cache) + (size_t)layer * layer_elems;
  aa.qpack = static_cast<__nv_bfloat16 *>(workspace);
  aa.status = status;
  const int t_slots = std::max(max_inline, (pl.R_pad + pl.G - 1) / pl.G);
  if (t_slots > INT32_MAX / 2 || batch > 65535)
    return fail(PIC_ERR_UNSUPPORTED, "%s: grid too large", who);
  dim3 agrid(t_slots, batch);
  cudaError_t le = D == 128 ? launch_dependent(append_kernel<128>, agrid, dim3(256), 0, stream, aa, rp)
                            : launch_dependent(append_kernel<64>, agrid, dim3(256), 0, stream, aa, rp);
  if (le != cudaSuccess) return cuda_fail(le, "append launch");
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "append launch");
  return PIC_OK;
}

// The inline projections of a prefill call: all three or none.
static pic_status_t check_projections(const char *who, const void *q, const void *k_new,
                                      const void *v_new) {
  const int given = (q != nullptr) + (k_new != nullptr) + (v_new != nullptr);
  if (given != 0 && given != 3)
    return fail(PIC_ERR_INVALID_ARG, "%s: give q, k_new and v_new together, or none", who);
  return PIC_OK;
}

}  // namespace prefill
}  // namespace pic

extern "C" pic_status_t pic_append_inline(
    const pic_geom_t *geom, int32_t layer, int32_t batch, int32_t max_inline, const void *q,
    const void *k_new, const void *v_new, const int32_t *inline_pos, const int32_t *inline_len,
    const int64_t *slot_mapping, int32_t max_ctx, int64_t num_pages, void *k_cache,
    void *v_cache, void *workspace, size_t workspace_bytes, pic_stream_t stream) {
  using namespace pic;
  using namespace pic::prefill;
  RopeParams rp;
  Plan pl;
  // the packed queries are the leading part of the prefill workspace (size of num_splits = 1)
  pic_status_t st = check_common("pic_append_inline", geom, layer, batch, max_inline, max_ctx,
                                 num_pages, 1, workspace, workspace_bytes, &rp, &pl);
  if (st != PIC_OK) return st;
  if (!q || !k_new || !v_new || !inline_pos || !inline_len || !slot_mapping || !k_cache ||
      !v_cache)
    return fail(PIC_ERR_INVALID_ARG, "pic_append_inline: NULL tensor");
  return launch_append("pic_append_inline", geom, rp, pl, layer, batch, max_inline, q, k_new,
                       v_new, inline_pos, inline_len, slot_mapping, nullptr, 0, max_ctx,
                       num_pages, k_cache, v_cache, workspace, stream);
}

namespace pic {
namespace prefill {

// The attention launch (and the merge launch when the key range is split).
template <int D, bool kFused>
static cudaError_t launch_attention(const Plan &pl, const Params &pp, const FusedArgs &fa,
                                    const RopeParams &rp, const CUtensorMap &tq,
                                    const CUtensorMap &tk, const CUtensorMap &tv,
                                    const CUtensorMap &tkp, const CUtensorMap &tvp,
                                    cudaStream_t stream) {
  const int smem = Layout<D>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<D, kFused>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  if constexpr (kFused) {
    // setmaxnreg.inc waits for registers the CTA was launched with: refuse to
    // launch a build whose register count at launch would not cover the split
    cudaFuncAttributes fa_attr;
    e = cudaFuncGetAttributes(&fa_attr, attn_kernel<D, kFused>);
    if (e != cudaSuccess) return e;
    if (fa_attr.numRegs < kRegLaunchFused) return cudaErrorInvalidConfiguration;
    // page sources and document cos/sin of the call, ahead of the attention
    const int page_blocks = (fa.n_pidx + 7) / 8;
    const int doc_blocks = (fa.max_docs + 256 / fa.half - 1) / (256 / fa.half);
    e = launch_dependent(fused_setup_kernel, dim3(page_blocks + doc_blocks, pp.batch), dim3(256), 0,
                         stream, fa, rp, pp.batch, page_blocks, pp.status);
    if (e != cudaSuccess) return e;
  }
  const int npairs = (pl.m_tiles + NQ - 1) / NQ;
  if constexpr (kFused) {
    // clusters of two consecutive query pairs: an even count per key split
    dim3 grid(((npairs + 1) & ~1) * pl.splits, pp.Hkv, pp.batch);
    e = launch_dependent_cluster(attn_kernel<D, kFused>, grid, dim3(threads_of<kFused>()), smem,
                                 stream, 2, tq, tk, tv, tkp, tvp, pp, fa, rp);
  } else {
    dim3 grid(npairs * pl.splits, pp.Hkv, pp.batch);
    e = launch_dependent(attn_kernel<D, kFused>, grid, dim3(threads_of<kFused>()), smem, stream,
                         tq, tk, tv, tkp, tvp, pp, fa, rp);
  }
  if (e != cudaSuccess) return e;
  if (pl.splits > 1) {
    const long long rows = (long long)pp.batch * pp.Hkv * pl.m_tiles * BM;
    e = launch_combine<D>(rows, pp, stream);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

}  // namespace prefill
}  // namespace pic

extern "C" pic_status_t pic_attend_prefill(
    const pic_geom_t *geom, int32_t layer, int32_t batch, int32_t max_inline, const void *q,
    const void *k_new, const void *v_new, const int32_t *inline_pos, const int32_t *inline_len,
    int32_t max_ctx, const int32_t *block_table, int32_t max_pages, int64_t num_pages,
    void *k_cache, void *v_cache, void *out, float *lse, int32_t num_splits, void *workspace,
    size_t workspace_bytes, pic_stream_t stream) {
  using namespace pic;
  using namespace pic::prefill;
  RopeParams rp;
  Plan pl;
  pic_status_t st = check_common("pic_attend_prefill", geom, layer, batch, max_inline, max_ctx,
                                 num_pages, num_splits, workspace, workspace_bytes, &rp, &pl);
  if (st != PIC_OK) return st;
  if (max_pages <= 0) return fail(PIC_ERR_INVALID_ARG, "pic_attend_prefill: max_pages <= 0");
  if (!inline_pos || !inline_len || !block_table || !k_cache || !v_cache || !out)
    return fail(PIC_ERR_INVALID_ARG, "pic_attend_prefill: NULL tensor");
  st = check_projections("pic_attend_prefill", q, k_new, v_new);
  if (st != PIC_OK) return st;
  // out may be page-locked host memory: the kernels then store the rows there
  out = device_address(out);
  if (!out)
    return fail(PIC_ERR_INVALID_ARG,
                "pic_attend_prefill: out is neither memory of the current device nor page-locked host memory");
  if ((reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache) |
       reinterpret_cast<uintptr_t>(out)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_attend_prefill: bf16 tensors must be 16-byte aligned");
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_attend_prefill: no device status word");
  if (q) {  // the inline tokens' RoPE and append first (slots from the block table)
    st = launch_append("pic_attend_prefill", geom, rp, pl, layer, batch, max_inline, q, k_new,
                       v_new, inline_pos, inline_len, nullptr, block_table, max_pages, max_ctx,
                       num_pages, k_cache, v_cache, workspace, stream);
    if (st != PIC_OK) return st;
  }
  const int D = geom->head_dim, Hkv = geom->num_kv_heads;
  const long long rows_total = (long long)geom->num_layers * num_pages * Hkv * 16;
  uint8_t *ws = static_cast<uint8_t *>(workspace);

  CUtensorMap tq, tk, tv;
  st = encode_tmap_2d(&tq, ws, D, (uint64_t)batch * Hkv * pl.R_pad, (uint64_t)D * 2, 64, BM);
  if (D == 128) {
    if (st == PIC_OK) st = encode_tmap_pages128(&tk, k_cache, (uint64_t)rows_total / 16);
    if (st == PIC_OK) st = encode_tmap_pages128(&tv, v_cache, (uint64_t)rows_total / 16);
  } else {
    if (st == PIC_OK) st = encode_tmap_2d(&tk, k_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
    if (st == PIC_OK) st = encode_tmap_2d(&tv, v_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
  }
  if (st != PIC_OK) return st;
  Params pp;
  pp.batch = batch;
  pp.Hq = geom->num_q_heads;
  pp.Hkv = Hkv;
  pp.G = pl.G;
  pp.max_inline = max_inline;
  pp.R_pad = pl.R_pad;
  pp.m_tiles = pl.m_tiles;
  pp.num_splits = pl.splits;
  pp.max_pages = max_pages;
  pp.oob_row = (int)rows_total;
  pp.num_pages = num_pages;
  pp.layer_row0 = (long long)layer * num_pages * Hkv * 16;
  pp.inline_pos = inline_pos;
  pp.inline_len = inline_len;
  pp.block_table = block_table;
  pp.out = static_cast<__nv_bfloat16 *>(out);
  pp.lse = lse;
  pp.part_o = pl.splits > 1 ? reinterpret_cast<__half *>(ws + pl.q_bytes) : nullptr;
  pp.part_ml = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes + pl.po_bytes) : nullptr;
  pp.status = status;
  pp.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D));

  cudaError_t e = D == 128 ? launch_attention<128, false>(pl, pp, FusedArgs{}, rp, tq, tk, tv, tk, tv, stream)
                           : launch_attention<64, false>(pl, pp, FusedArgs{}, rp, tq, tk, tv, tk, tv, stream);
  if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill launch");
  return PIC_OK;
}

extern "C" pic_status_t pic_attend_prefill_fused(
    const pic_geom_t *geom, int32_t layer, int32_t batch, int32_t max_inline, const void *q,
    const void *k_new, const void *v_new, const int32_t *inline_pos, const int32_t *inline_len,
    int32_t max_ctx, const int32_t *block_table, int32_t max_pages, int64_t num_pages,
    void *k_cache, void *v_cache, const void *k_pool, const void *v_pool, int64_t pool_tokens,
    int32_t max_docs, const int64_t *tok_map, const int32_t *doc_delta, void *out, float *lse,
    int32_t num_splits, void *workspace, size_t workspace_bytes, pic_stream_t stream) {
  using namespace pic;
  using namespace pic::prefill;
  static const char *who = "pic_attend_prefill_fused";
  RopeParams rp;
  Plan pl;
  pic_status_t st = check_common(who, geom, layer, batch, max_inline, max_ctx, num_pages,
                                 num_splits, workspace, workspace_bytes, &rp, &pl);
  if (st != PIC_OK) return st;
  if (max_pages <= 0 || pool_tokens <= 0 || max_docs < 0)
    return fail(PIC_ERR_INVALID_ARG, "%s: sizes must be positive", who);
  if (max_docs > 65535 * 256)
    return fail(PIC_ERR_UNSUPPORTED, "%s: max_docs too large", who);
  const size_t ws_need = pl.total + fused_page_bytes(pl, batch) + fused_cs_bytes(geom, batch, max_docs);
  if (workspace_bytes < ws_need)
    return fail(PIC_ERR_WORKSPACE, "%s: workspace needs %zu bytes (pic_prefill_fused_workspace_size)",
                who, ws_need);
  if ((long long)geom->num_layers * pool_tokens >= (long long)INT32_MAX)
    return fail(PIC_ERR_UNSUPPORTED, "%s: pool has more than 2^31 rows", who);
  if (!inline_pos || !inline_len || !block_table || !k_cache || !v_cache || !k_pool || !v_pool ||
      !out || !tok_map || (max_docs > 0 && !doc_delta))
    return fail(PIC_ERR_INVALID_ARG, "%s: NULL tensor", who);
  st = check_projections(who, q, k_new, v_new);
  if (st != PIC_OK) return st;
  out = device_address(out);
  if (!out)
    return fail(PIC_ERR_INVALID_ARG,
                "%s: out is neither memory of the current device nor page-locked host memory", who);
  if ((reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache) |
       reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
       reinterpret_cast<uintptr_t>(out)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "%s: bf16 tensors must be 16-byte aligned", who);
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "%s: no device status word", who);
  if (q) {  // the inline tokens' RoPE and append first (slots from the block table)
    st = launch_append(who, geom, rp, pl, layer, batch, max_inline, q, k_new, v_new, inline_pos,
                       inline_len, nullptr, block_table, max_pages, max_ctx, num_pages, k_cache,
                       v_cache, workspace, stream);
    if (st != PIC_OK) return st;
  }
  const int D = geom->head_dim, Hkv = geom->num_kv_heads;
  const long long rows_total = (long long)geom->num_layers * num_pages * Hkv * 16;
  const uint64_t pool_rows = (uint64_t)geom->num_layers * pool_tokens;
  uint8_t *ws = static_cast<uint8_t *>(workspace);

  CUtensorMap tq, tk, tv, tkp, tvp;
  st = encode_tmap_2d(&tq, ws, D, (uint64_t)batch * Hkv * pl.R_pad, (uint64_t)D * 2, 64, BM);
  const bool pool_boxes = pool_rows > 16;  // else the maps below are placeholders, never used
  if (D == 128) {
    if (st == PIC_OK) st = encode_tmap_pages128(&tk, k_cache, (uint64_t)rows_total / 16);
    if (st == PIC_OK) st = encode_tmap_pages128(&tv, v_cache, (uint64_t)rows_total / 16);
    if (st == PIC_OK) st = encode_tmap_pool128(&tkp, k_pool, pool_boxes ? pool_rows : 17, Hkv);
    if (st == PIC_OK) st = encode_tmap_pool128(&tvp, v_pool, pool_boxes ? pool_rows : 17, Hkv);
  } else {
    if (st == PIC_OK) st = encode_tmap_2d(&tk, k_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
    if (st == PIC_OK) st = encode_tmap_2d(&tv, v_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
    if (st == PIC_OK)
      st = encode_tmap_3d(&tkp, k_pool, D, Hkv, pool_boxes ? pool_rows : 16, (uint64_t)D * 2,
                          (uint64_t)Hkv * D * 2, 64, 1, 16);
    if (st == PIC_OK)
      st = encode_tmap_3d(&tvp, v_pool, D, Hkv, pool_boxes ? pool_rows : 16, (uint64_t)D * 2,
                          (uint64_t)Hkv * D * 2, 64, 1, 16);
  }
  if (st != PIC_OK) return st;

  Params pp;
  pp.batch = batch;
  pp.Hq = geom->num_q_heads;
  pp.Hkv = Hkv;
  pp.G = pl.G;
  pp.max_inline = max_inline;
  pp.R_pad = pl.R_pad;
  pp.m_tiles = pl.m_tiles;
  pp.num_splits = pl.splits;
  pp.max_pages = max_pages;
  pp.oob_row = (int)rows_total;
  pp.num_pages = num_pages;
  pp.layer_row0 = (long long)layer * num_pages * Hkv * 16;
  pp.inline_pos = inline_pos;
  pp.inline_len = inline_len;
  pp.block_table = block_table;
  pp.out = static_cast<__nv_bfloat16 *>(out);
  pp.lse = lse;
  pp.part_o = pl.splits > 1 ? reinterpret_cast<__half *>(ws + pl.q_bytes) : nullptr;
  pp.part_ml = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes + pl.po_bytes) : nullptr;
  pp.status = status;
  pp.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D));
  FusedArgs fa;
  fa.tok_map = tok_map;
  fa.doc_delta = doc_delta;
  fa.k_pool = static_cast<const __nv_bfloat16 *>(k_pool);
  fa.v_pool = static_cast<const __nv_bfloat16 *>(v_pool);
  fa.k_cache = static_cast<const __nv_bfloat16 *>(k_cache);
  fa.v_cache = static_cast<const __nv_bfloat16 *>(v_cache);
  fa.pool_tokens = pool_tokens;
  fa.max_ctx = max_ctx;
  fa.max_docs = max_docs;
  fa.layer = layer;
  fa.pool_boxes = pool_boxes;
  fa.page_src = reinterpret_cast<const PageSrcEntry *>(ws + pl.total);
  fa.doc_cs = reinterpret_cast<const float2 *>(ws + pl.total + fused_page_bytes(pl, batch));
  fa.n_pidx = pl.n_pidx;
  fa.half = D / 2;
  cudaError_t e = D == 128 ? launch_attention<128, true>(pl, pp, fa, rp, tq, tk, tv, tkp, tvp, stream)
                           : launch_attention<64, true>(pl, pp, fa, rp, tq, tk, tv, tkp, tvp, stream);
  if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill_fused launch");
  return PIC_OK;
}
