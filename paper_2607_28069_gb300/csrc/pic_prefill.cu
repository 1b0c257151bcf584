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
#include "pic_internal.cuh"

namespace pic {
namespace prefill {

constexpr int BM = 128;  // query rows per tile (TMEM lanes)
constexpr int NQ = 2;    // query tiles per CTA, sharing every K/V tile
constexpr int BN = 128;  // keys per KV tile
constexpr int NSK = 3;   // K ring stages (released after the last QK of a tile)
constexpr int NSV = 2;   // V ring stages (released after the last PV of a tile)
constexpr int kThreads = 128 + NQ * 128;  // K producer, MMA, NQ softmax warpgroups, V producer, relay
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
  static constexpr int kBytes = kBar + 256;
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
  B_COUNT = B_OFINAL + 1
};

struct Params {
  int batch, Hq, Hkv, G, max_inline, R_pad, m_tiles, num_splits, max_pages, oob_row;
  long long num_pages, layer_row0;
  const int32_t *inline_pos, *inline_len, *block_table;
  __nv_bfloat16 *out;
  float *lse, *part_o, *part_ml;
  int32_t *status;
  float scale_log2;
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
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                const __grid_constant__ CUtensorMap tm_v, Params p) {
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
  // Grid (split + splits * pair, kv head, request), pairs in reverse order.
  // CTAs start in linear block order, so all CTAs of one (request, kv head)
  // start together and its K/V, read by every pair, is reused from L2; within
  // the group the pairs of the last query rows, which see the most keys, go
  // first and the short prefix-row pairs fill in behind them.
  const int npairs = (int)gridDim.x / p.num_splits;
  const int split = blockIdx.x % p.num_splits;
  const int pair = npairs - 1 - (int)blockIdx.x / p.num_splits;
  const int hk = blockIdx.y, b = blockIdx.z;
  const int detail = b;

  // ---- set-up that reads nothing the previous kernel writes: it runs before
  // the programmatic-launch wait, while that kernel may still be finishing
  if (threadIdx.x == 0) {
    for (int i = 0; i < B_COUNT; ++i)
      mbar_init(bar(i), (i >= B_PFULL && i < B_PFULL + NQ) ? 4 : 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_q);
    prefetch_tmap(&tm_k);
    prefetch_tmap(&tm_v);
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
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
  int r0[NQ], kmin[NQ], kmax[NQ], ntile = 0;
#pragma unroll
  for (int t = 0; t < NQ; ++t) {
    r0[t] = (pair * NQ + t) * BM;
    kmin[t] = kmax[t] = -1;
    if (r0[t] < rows && t < p.m_tiles - pair * NQ) {
      kmin[t] = ipos[r0[t] / p.G];
      kmax[t] = ipos[(min(r0[t] + BM, rows) - 1) / p.G];
      ntile = t + 1;
    }
  }
  if (ntile == 0) {  // no query row in this pair
    release_and_exit();
    return;
  }
  const int kmax_all = ntile == 2 ? kmax[1] : kmax[0];
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

  if (warp == 0 || warp == kWarpV) {
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
  } else if (warp == 1) {
    // ===================================================== MMA issuer
    // The whole warp takes part in the named barriers; lane 0 issues.  After
    // an abort both this loop and the relay's run to the end (skipping their
    // waits and MMAs), so every barrier sync has its arrival.
    const bool leader = lane == 0;
    if (leader) mbar_wait(bar(B_Q), 0, abort_flag, p.status, detail);
    __syncwarp();
    tc_fence_after();
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
            if (t == ntile - 1) mma_commit(bar(B_VEMPTY + pst));  // last reader of V(j-1)
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
            if (t == ntile - 1) mma_commit(bar(B_KEMPTY + st));  // last reader of K(j)
          }
        }
      }
    }
    if (leader) mma_commit(bar(B_OFINAL));
  } else if (warp == kWarpRelay) {
    // ===================================================== relay for the issuer
    // Mirrors the issuer's loop: the same conditions, the same order.  Its
    // arrival on a barrier in iteration j + 1 depends on an MMA the issuer
    // issues only after its sync on that barrier in iteration j, so the two
    // never get a phase apart.
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
          mbar_wait(bar(B_KFULL + j % NSK), (j / NSK) & 1, abort_flag, p.status, detail);
          named_bar_arrive(kNbK, 64);
          k_ready = true;
        }
      }
    }
  } else {
    // ===================================================== softmax warpgroups
    static_assert(NQ == 2, "softmax warpgroup selection assumes two query tiles");
    const int t = (warp - 2) >> 2;  // query tile of this warpgroup
    const int wq = warp & 3;        // TMEM lane quarter
    const int row = wq * 32 + lane;
    // constant-index selects keep the per-tile values in registers
    const int my_r0 = t == 0 ? r0[0] : r0[1];
    const int my_kmin = t == 0 ? kmin[0] : kmin[1];
    const int my_n = t < ntile ? (t == 0 ? nt[0] : nt[1]) : 0;
    const size_t my_part0 = part_row0(t);
    const int rg = my_r0 + row;
    const bool valid = t < ntile && rg < rows;
    const int tok = rg / p.G, g = rg % p.G;
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
      // row max: 4 independent chains of 3-input max
      float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int c = 0; c < BN; c += 8)
#pragma unroll
        for (int i = 0; i < 4; ++i) mx[i] = max3f(mx[i], s[c + 2 * i], s[c + 2 * i + 1]);
      const float m_new = fmaxf(m_used, max3f(mx[0], mx[1], fmaxf(mx[2], mx[3])) * p.scale_log2);
      float alpha = 1.f;
      const bool resc = m_new > m_used + 8.f;
      if (resc) {
        alpha = ex2(m_used - m_new);
        m_used = m_new;
      }
      const float mref = (m_used == -INFINITY) ? 0.f : m_used;
      // P = exp2(s * scale - m) as bf16, written over S in 16-column chunks as
      // soon as each 32-key chunk is done (S was read completely above, so the
      // overlap is harmless and the packed values never pile up in registers).
      // Scaling and the row sum run on packed fp32 pairs (half the issue
      // slots; the softmax is bound by instruction issue, not by MUFU).
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
      float l0, l1;
      f2unpack(acc[0], l0, l1);
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
      constexpr int kRowOut = D * 2 + 16, kRowPart = D * 4 + 16;
      uint8_t *stage = smem + (size_t)t * BM * (single ? kRowOut : kRowPart);
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
          float4 *dst = reinterpret_cast<float4 *>(stage + row * kRowPart);
#pragma unroll
          for (int q = 0; q < D / 4; ++q)
            dst[q] = make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
          p.part_ml[(my_part0 + row) * 2] = (l > 0.f) ? m_used : -INFINITY;
          p.part_ml[(my_part0 + row) * 2 + 1] = l;
        }
      }
      asm volatile("bar.sync %0, 128;" ::"r"(1 + t) : "memory");
      if (ok) {
        const int nrows = min(BM, rows - my_r0);  // valid rows of this tile
        if (single) {
          // 16 lanes per 256-byte row (D = 128) or 8 per 128-byte row (D = 64)
          constexpr int LPR = D / 8, RPI = 32 / LPR;
          for (int r = wq * RPI + lane / LPR; r < nrows; r += 4 * RPI) {
            const int rg2 = my_r0 + r, tk = rg2 / p.G, gg = rg2 % p.G;
            const uint4 v = *reinterpret_cast<const uint4 *>(stage + r * kRowOut + (lane % LPR) * 16);
            st_global16(p.out + (((size_t)b * p.max_inline + tk) * p.Hq + hk * p.G + gg) * D +
                            (lane % LPR) * 8, v);
          }
        } else {
          // fp32 rows are contiguous in the partial buffer: one row per warp pass
          constexpr int LPR = D / 4;  // 16-byte pieces per row
          constexpr int RPI = 32 / LPR > 0 ? 32 / LPR : 1;
          for (int r = wq * RPI + lane / LPR; r < nrows; r += 4 * RPI)
#pragma unroll
            for (int c = lane % LPR; c < D / 4; c += (LPR < 32 ? LPR : 32)) {
              const float4 v = *reinterpret_cast<const float4 *>(stage + r * kRowPart + c * 16);
              reinterpret_cast<float4 *>(p.part_o + (my_part0 + r) * D)[c] = v;
            }
        }
      }
    }
  }
  // Release the dependent launch (the split merge, or the next layer's
  // append) only now: released at the start, it made the pass slower.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  tc_fence_before();
  __syncthreads();
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

// ===========================================================================
// Fused rotate-on-load prefill attention (documents read from the pool).
//
// Instead of reading relocated keys R(delta_k) k from the stitched cache, the
// kernel reads the documents' keys and values straight from the pool (as they
// were compiled) and rotates the *queries* the other way:
//     (R(p) q) . (R(delta_k) k) = (R(-delta_k) R(p) q) . k,
// since rotations are orthogonal.  Per document the query tile is turned into
// Q'_k = R(-delta_k) Q in TMEM by the softmax threads (each owns one TMEM lane,
// i.e. one query row) and the QK^T MMA takes its A operand from TMEM.  Prefix
// and query keys (written by pic_append_inline) still come from the paged
// cache.  A pool tile is 128 consecutive rows of one document: two 16 KB TMA
// boxes per operand instead of 16 page boxes.
//
// Key tiles are segment aligned: the prefix [0, P) and the query span [Q0, Q1)
// in 128-key tiles of the absolute position grid (keys outside the segment
// masked), each document in 128-key tiles from its first token (keys past its
// end masked).  Everything else (splits, pipeline, epilogue) is as in
// attn_kernel's single-tile form.
// TMEM: S_0 [0,128), S_1 [128,256), O [256,256+D), Q'_0 [384,384+D/2),
// Q'_1 [448,448+D/2) (bf16 pairs).
namespace fused {

constexpr int BN = 128, NST = 2, kThreads = 192, kMaxDocs = 1024;

template <int D>
struct Layout {
  static constexpr int kTile = BN * D * 2;
  static constexpr int kQ = 0;
  static constexpr int kK = kQ + BM * D * 2;
  static constexpr int kV = kK + NST * kTile;
  static constexpr int kMeta = kV + NST * kTile;
  // seg_first[2 kMaxDocs + 2] int32, off/len/delta [kMaxDocs] int32, start [kMaxDocs] int64
  static constexpr int kSegFirst = kMeta;
  static constexpr int kOff = kSegFirst + (2 * kMaxDocs + 4) * 4;
  static constexpr int kLen = kOff + kMaxDocs * 4;
  static constexpr int kDelta = kLen + kMaxDocs * 4;
  static constexpr int kStart = kDelta + kMaxDocs * 4;
  static constexpr int kCS = kStart + kMaxDocs * 8;  // 64 float2
  static constexpr int kBar = kCS + 64 * 8;
  static constexpr int kBytes = kBar + 256;
  static constexpr int kAlloc = kBytes + 1024;
};

enum {
  F_Q = 0,
  F_KFULL = 1,
  F_VFULL = F_KFULL + NST,
  F_KVEMPTY = F_VFULL + NST,
  F_SFULL = F_KVEMPTY + NST,
  F_PFULL = F_SFULL + 2,
  F_PFREE = F_PFULL + 2,
  F_QREADY = F_PFREE + 2,
  F_OFINAL = F_QREADY + 2,
  F_COUNT = F_OFINAL + 1
};

struct FParams {
  Params base;
  RopeParams rp;
  long long pool_tokens;
  int max_docs, layer;
  const int32_t *num_docs, *doc_offset, *doc_delta, *ids, *doc_len;
  const int64_t *doc_start;
};

// The tile sequence seen by every role.  Segment s: 0 = prefix, 1..m = doc
// s-1, m+1 = query.  seg_first[s] = index of the segment's first tile.
struct TileInfo {
  int doc;         // document index, -1 for a cache tile
  int key_base;    // logical position of smem row 0
  int vlo, vhi;    // valid logical key range of this tile
  int cache_kt;    // absolute 128-key tile index (cache tiles)
  long long prow;  // pool row of smem row 0 (document tiles)
  bool doc_first;  // first tile of its document
};

// Segments of a query tile's visible keys in logical order: cache segment
// C_0 (the prefix), document D_0, C_1 (the inline span after D_0), D_1, ...,
// D_{m-1}, C_m (the last span and the query).  Segment 2c is C_c, 2k+1 is
// D_k; every range is clipped to the keys below kend.
struct Seq {
  const int32_t *seg_first, *off, *len, *delta;
  const long long *start;
  int m, kend;
  __device__ int cache_lo(int c) const { return c == 0 ? 0 : min(off[c - 1] + len[c - 1], kend); }
  __device__ int cache_hi(int c) const { return c < m ? min(off[c], kend) : kend; }
  __device__ TileInfo at(int t) const {
    // segment containing global tile t (binary search over seg_first[0..2m+1))
    int lo = 0, hi = 2 * m;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (seg_first[mid] <= t) lo = mid;
      else hi = mid - 1;
    }
    const int j = t - seg_first[lo];
    TileInfo ti;
    if ((lo & 1) == 0) {
      const int a = cache_lo(lo >> 1), e = cache_hi(lo >> 1);
      ti.doc = -1;
      ti.cache_kt = a / BN + j;
      ti.key_base = ti.cache_kt * BN;
      ti.vlo = max(a, ti.key_base);
      ti.vhi = min(e, ti.key_base + BN);
      ti.prow = 0;
      ti.doc_first = false;
    } else {
      const int k = lo >> 1;
      ti.doc = k;
      ti.cache_kt = -1;
      ti.key_base = off[k] + j * BN;
      ti.vlo = ti.key_base;
      ti.vhi = min(off[k] + len[k], ti.key_base + BN);
      ti.prow = start[k] + (long long)j * BN;
      ti.doc_first = j == 0;
    }
    return ti;
  }
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_fused_kernel(const __grid_constant__ CUtensorMap tm_q,
                      const __grid_constant__ CUtensorMap tm_k,
                      const __grid_constant__ CUtensorMap tm_v,
                      const __grid_constant__ CUtensorMap tm_kp,
                      const __grid_constant__ CUtensorMap tm_vp, FParams fp) {
  // programmatic dependent launch: the kernel before (the append) has finished
  asm volatile("griddepcontrol.wait;" ::: "memory");
  using L = Layout<D>;
  const Params &p = fp.base;
  constexpr int PANELS = D / 64;
  constexpr uint32_t IDESC_QK = idesc_bf16(BM, BN, false, false);
  constexpr uint32_t IDESC_PV = idesc_bf16(BM, D, false, true);

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + L::kBar;
  auto bar = [&](int i) { return bar0 + 8u * (uint32_t)i; };
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + L::kBar + 8 * F_COUNT);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::kBar + 8 * F_COUNT + 8);
  int32_t *s_seg = reinterpret_cast<int32_t *>(smem + L::kSegFirst);
  int32_t *s_off = reinterpret_cast<int32_t *>(smem + L::kOff);
  int32_t *s_len = reinterpret_cast<int32_t *>(smem + L::kLen);
  int32_t *s_delta = reinterpret_cast<int32_t *>(smem + L::kDelta);
  long long *s_start = reinterpret_cast<long long *>(smem + L::kStart);
  float2 *s_cs = reinterpret_cast<float2 *>(smem + L::kCS);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x / p.num_splits, split = blockIdx.x % p.num_splits;
  const int hk = blockIdx.y, b = blockIdx.z;
  const int detail = b;

  const int tin = min(max(p.inline_len[b], 0), p.max_inline);
  const int rows = tin * p.G;
  const int r0 = mt * BM;
  if (r0 >= rows) return;
  const int r_last = min(r0 + BM, rows) - 1;
  const int32_t *ipos = p.inline_pos + (size_t)b * p.max_inline;
  const int kmax = ipos[r_last / p.G];

  // ---- per-document metadata into shared memory (all threads)
  const int m = min(max(fp.num_docs[b], 0), fp.max_docs);
  for (int k = threadIdx.x; k < m; k += kThreads) {
    const size_t i = (size_t)b * fp.max_docs + k;
    const int id = fp.ids[i];
    s_off[k] = fp.doc_offset[i];
    s_delta[k] = fp.doc_delta[i];
    s_len[k] = (id >= 0) ? fp.doc_len[id] : 0;
    s_start[k] = (id >= 0) ? fp.doc_start[id] : 0;
  }
  __syncthreads();
  Seq sq;
  sq.seg_first = s_seg;
  sq.off = s_off;
  sq.len = s_len;
  sq.delta = s_delta;
  sq.start = s_start;
  sq.m = m;
  sq.kend = kmax + 1;  // keys at or beyond kend are never visible here
  if (threadIdx.x == 0) {  // tiles per segment, prefix sums (m <= kMaxDocs, serial is fine)
    int t = 0;
    auto cache_tiles = [&](int a, int e) { return e > a ? (e - 1) / BN - a / BN + 1 : 0; };
    for (int c = 0; c <= m; ++c) {
      s_seg[2 * c] = t;
      t += cache_tiles(sq.cache_lo(c), sq.cache_hi(c));
      if (c == m) break;
      s_seg[2 * c + 1] = t;
      const int e = min(s_off[c] + s_len[c], sq.kend);
      t += e > s_off[c] ? (e - s_off[c] + BN - 1) / BN : 0;
    }
    s_seg[2 * m + 1] = t;
  }
  __syncthreads();
  const int n_all = s_seg[2 * m + 1];
  const int per = (n_all + p.num_splits - 1) / p.num_splits;
  const int kv_begin = split * per;
  const int n = max(0, min(per, n_all - kv_begin));
  const size_t part_row0 =
      ((((size_t)b * p.Hkv + hk) * p.m_tiles + mt) * p.num_splits + split) * BM;
  if (n == 0) {
    if (p.num_splits > 1 && threadIdx.x < BM) {
      p.part_ml[(part_row0 + threadIdx.x) * 2] = -INFINITY;
      p.part_ml[(part_row0 + threadIdx.x) * 2 + 1] = 0.f;
    }
    return;
  }

  if (threadIdx.x == 0) {
    for (int i = 0; i < F_COUNT; ++i)
      mbar_init(bar(i), (i == F_PFULL || i == F_PFULL + 1 || i == F_QREADY || i == F_QREADY + 1)
                            ? 128 : 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = *tmem_slot;

  if (warp == 0) {
    // ===================================================== TMA producer
    const int32_t *bt = p.block_table + (size_t)b * p.max_pages;
    if (lane == 0) {
      prefetch_tmap(&tm_q);
      prefetch_tmap(&tm_k);
      prefetch_tmap(&tm_v);
      prefetch_tmap(&tm_kp);
      prefetch_tmap(&tm_vp);
      mbar_expect_tx(bar(F_Q), BM * D * 2);
      const int qrow = (b * p.Hkv + hk) * p.R_pad + r0;
      for (int pn = 0; pn < PANELS; ++pn)
        tma_load_2d(sbase + L::kQ + pn * BM * 128, &tm_q, pn * 64, qrow, bar(F_Q));
    }
    int issued = 0;
    for (int j = 0; j < n; ++j) {
      const int st = j % NST;
      const TileInfo ti = sq.at(kv_begin + j);
      int y = p.oob_row;  // cache tile: lanes 0..7 look up their page
      if (ti.doc < 0 && lane < 8) {
        const int pidx = ti.cache_kt * 8 + lane;
        if (pidx * 16 < ti.vhi && pidx < p.max_pages) {
          const int page = bt[pidx];
          if (page >= 0 && page < p.num_pages)
            y = (int)(p.layer_row0 + ((long long)page * p.Hkv + hk) * 16);
          else
            dev_fail(p.status, PIC_DEV_BAD_PAGE, detail);
        }
      }
      if (j >= NST) {
        const bool ok = mbar_wait(bar(F_KVEMPTY + st), ((j / NST) - 1) & 1, abort_flag, p.status, detail);
        if (!__all_sync(0xffffffffu, ok)) break;
      }
      if (lane == 0) mbar_expect_tx(bar(F_KFULL + st), L::kTile);
      if (lane == 16) mbar_expect_tx(bar(F_VFULL + st), L::kTile);
      __syncwarp();
      if (ti.doc < 0) {
        const int box = lane & 15, bpage = box / PANELS, bpanel = box % PANELS;
        const int yb = __shfl_sync(0xffffffffu, y, bpage);
        if (box < 8 * PANELS) {
          const uint32_t off = st * L::kTile + bpanel * BN * 128 + bpage * 16 * 128;
          if (lane < 16)
            tma_load_2d(sbase + L::kK + off, &tm_k, bpanel * 64, yb, bar(F_KFULL + st));
          else
            tma_load_2d(sbase + L::kV + off, &tm_v, bpanel * 64, yb, bar(F_VFULL + st));
        }
      } else {
        // two 128-row boxes per operand, straight from the pool rows of the document
        const int z = (int)((long long)fp.layer * fp.pool_tokens + ti.prow);
        if (lane < PANELS)
          tma_load_3d(sbase + L::kK + st * L::kTile + lane * BN * 128, &tm_kp, lane * 64, hk, z,
                      bar(F_KFULL + st));
        else if (lane >= 16 && lane < 16 + PANELS)
          tma_load_3d(sbase + L::kV + st * L::kTile + (lane - 16) * BN * 128, &tm_vp,
                      (lane - 16) * 64, hk, z, bar(F_VFULL + st));
      }
      issued = j + 1;
    }
    if (lane == 0 && *abort_flag) {
      for (int j = max(0, issued - NST); j < issued; ++j) {
        mbar_wait(bar(F_KFULL + j % NST), (j / NST) & 1, abort_flag, p.status, detail);
        mbar_wait(bar(F_VFULL + j % NST), (j / NST) & 1, abort_flag, p.status, detail);
      }
    }
  } else if (warp == 1) {
    // ===================================================== MMA issuer
    if (lane == 0) {
      const uint32_t tS0 = tbase, tO = tbase + 256, tQd = tbase + 384;
      bool ok = mbar_wait(bar(F_Q), 0, abort_flag, p.status, detail);
      tc_fence_after();
      // base descriptors; stages and k-steps add (offset >> 4) to the address field
      const uint64_t dQ = sdesc_sw128(sbase + L::kQ, 16, 1024);
      const uint64_t dK = sdesc_sw128(sbase + L::kK, 16, 1024);
      const uint64_t dV = sdesc_sw128(sbase + L::kV, BN * 128, 1024);
      int dcount = -1;  // documents entered so far in this split
      for (int j = 0; ok && j <= n; ++j) {
        if (j < n) {
          const int st = j % NST, sb = j & 1;
          const TileInfo ti = sq.at(kv_begin + j);
          if (ti.doc >= 0 && (ti.doc_first || j == 0)) {  // entering a document
            ++dcount;
            if (!mbar_wait(bar(F_QREADY + (dcount & 1)), (dcount >> 1) & 1, abort_flag, p.status, detail)) break;
          }
          if (!mbar_wait(bar(F_KFULL + st), (j / NST) & 1, abort_flag, p.status, detail)) break;
          tc_fence_after();
          const uint64_t dk = dK + (uint64_t)((st * L::kTile) >> 4);
          if (ti.doc < 0) {
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              mma_ss(tS0 + sb * 128, dQ + ((kk >> 2) * (BM * 128) + (kk & 3) * 32) / 16,
                     dk + ((kk >> 2) * (BN * 128) + (kk & 3) * 32) / 16, IDESC_QK, kk > 0);
          } else {
            const uint32_t qa = tQd + (dcount & 1) * 64;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk)
              mma_ts(tS0 + sb * 128, qa + kk * 8, dk + ((kk >> 2) * (BN * 128) + (kk & 3) * 32) / 16,
                     IDESC_QK, kk > 0);
          }
          mma_commit(bar(F_SFULL + sb));
        }
        if (j >= 1) {
          const int pj = j - 1, pst = pj % NST, pb = pj & 1;
          if (!mbar_wait(bar(F_PFULL + pb), (pj >> 1) & 1, abort_flag, p.status, detail)) break;
          if (!mbar_wait(bar(F_VFULL + pst), (pj / NST) & 1, abort_flag, p.status, detail)) break;
          tc_fence_after();
          const uint64_t dv = dV + (uint64_t)((pst * L::kTile) >> 4);
#pragma unroll
          for (int kk = 0; kk < BN / 16; ++kk)
            mma_ts(tO, tS0 + pb * 128 + kk * 8, dv + (kk * 16 * 128) / 16, IDESC_PV,
                   (pj > 0 || kk > 0));
          mma_commit(bar(F_KVEMPTY + pst));
          mma_commit(bar(F_PFREE + pb));
        }
      }
      mma_commit(bar(F_OFINAL));
    }
  } else {
    // ===================================================== softmax warps
    const int wq = warp & 3;
    const int row = wq * 32 + lane;
    const int rg = r0 + row;
    const bool valid = rg < rows;
    const int tok = rg / p.G, g = rg % p.G;
    const int pos = valid ? ipos[tok] : -1;
    const uint32_t tl = tbase + ((uint32_t)(wq * 32) << 16);
    const uint32_t tQd = tl + 384;
    const int tid128 = threadIdx.x - 64;
    bool ok = true;

    float m_used = -INFINITY, l = 0.f;
    int dcount = -1;
    // Q'_k = R(-delta_k) Q for this thread's row, into TMEM buffer `buf`.
    auto make_qd = [&](int k, int buf) {
      asm volatile("bar.sync 1, 128;" ::: "memory");  // previous table no longer read
      if (tid128 < D / 2) {
        const float2 cs = rope_cos_sin(s_delta[k], rope_theta(fp.rp, fp.layer, tid128));
        s_cs[tid128] = make_float2(cs.x, -cs.y);  // R(-delta): sin changes sign
      }
      asm volatile("bar.sync 1, 128;" ::: "memory");
      // my row of Q from shared memory (128-byte swizzled panels), rotate, pack
      float x[D];
      const uint8_t *qs = smem + L::kQ;
#pragma unroll
      for (int c = 0; c < D / 8; ++c) {
        const int pn = c >> 3, ch = c & 7;
        const uint4 v = *reinterpret_cast<const uint4 *>(
            qs + pn * BM * 128 + row * 128 + ((ch ^ (row & 7)) << 4));
        unpack8(v, x + 8 * c);
      }
      uint32_t pk[D / 2];
      if (fp.rp.style == PIC_ROPE_HALF) {
#pragma unroll
        for (int i = 0; i < D / 2; ++i) {
          const float2 cs = s_cs[i];
          const float u = x[i], w = x[i + D / 2];
          x[i] = fmaf(u, cs.x, -w * cs.y);
          x[i + D / 2] = fmaf(u, cs.y, w * cs.x);
        }
      } else {
#pragma unroll
        for (int i = 0; i < D / 2; ++i) {
          const float2 cs = s_cs[i];
          const float u = x[2 * i], w = x[2 * i + 1];
          x[2 * i] = fmaf(u, cs.x, -w * cs.y);
          x[2 * i + 1] = fmaf(u, cs.y, w * cs.x);
        }
      }
#pragma unroll
      for (int i = 0; i < D / 2; ++i) pk[i] = pack2(x[2 * i], x[2 * i + 1]);
#pragma unroll
      for (int c = 0; c < D / 64; ++c) tmem_st32(tQd + buf * 64 + c * 32, pk + c * 32);
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(bar(F_QREADY + buf));
    };

    if (!__all_sync(0xffffffffu, mbar_wait(bar(F_Q), 0, abort_flag, p.status, detail))) ok = false;
    // documents of this split, in order: first one prepared up front
    int next_doc = -1;  // next document whose Q' is still to be prepared
    if (ok) {
      for (int j = 0; j < n; ++j) {
        const TileInfo ti = sq.at(kv_begin + j);
        if (ti.doc >= 0) {
          next_doc = ti.doc;
          break;
        }
      }
      if (next_doc >= 0) {
        make_qd(next_doc, 0);
        ++next_doc;
      }
    }
    int last_tile_doc = -1;  // last document with a tile in this split
    for (int j = n - 1; ok && j >= 0; --j) {
      const int dj = sq.at(kv_begin + j).doc;
      if (dj >= 0) {
        last_tile_doc = dj;
        break;
      }
    }
    for (int j = 0; ok && j < n; ++j) {
      const int sb = j & 1;
      const TileInfo ti = sq.at(kv_begin + j);
      if (!__all_sync(0xffffffffu, mbar_wait(bar(F_SFULL + sb), (j >> 1) & 1, abort_flag, p.status, detail))) {
        ok = false;
        break;
      }
      tc_fence_after();
      if (ti.doc >= 0 && (ti.doc_first || j == 0)) {
        ++dcount;
        // S of this document's first tile is ready, so every QK of the
        // document before it has finished: its Q' buffer may be reused.
        if (next_doc >= 0 && next_doc <= last_tile_doc) {
          make_qd(next_doc, (dcount + 1) & 1);
          ++next_doc;
        }
      }
      float s[BN];
#pragma unroll
      for (int c = 0; c < BN / 32; ++c)
        tmem_ld32(tl + sb * 128 + c * 32, reinterpret_cast<uint32_t *>(s + c * 32));
      tmem_wait_ld();
      {
        const int lo = ti.vlo - ti.key_base, hi = min(ti.vhi, pos + 1) - ti.key_base;
        if (lo > 0 || hi < BN) {
#pragma unroll
          for (int c = 0; c < BN; ++c)
            if (c < lo || c >= hi) s[c] = -INFINITY;
        }
      }
      float mx8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx8[i] = s[i];
#pragma unroll
      for (int c = 8; c < BN; c += 8)
#pragma unroll
        for (int i = 0; i < 8; ++i) mx8[i] = fmaxf(mx8[i], s[c + i]);
#pragma unroll
      for (int w = 4; w; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; ++i) mx8[i] = fmaxf(mx8[i], mx8[i + w]);
      const float m_new = fmaxf(m_used, mx8[0] * p.scale_log2);
      float alpha = 1.f;
      const bool resc = m_new > m_used + 8.f;
      if (resc) {
        alpha = ex2(m_used - m_new);
        m_used = m_new;
      }
      const float mref = (m_used == -INFINITY) ? 0.f : m_used;
      float ls8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) ls8[i] = 0.f;
      uint32_t pk[BN / 2];
#pragma unroll
      for (int c = 0; c < BN; c += 2) {
        const float p0 = ex2(fmaf(s[c], p.scale_log2, -mref));
        const float p1 = ex2(fmaf(s[c + 1], p.scale_log2, -mref));
        ls8[(c >> 1) & 7] += p0 + p1;
        pk[c / 2] = pack2(p0, p1);
      }
#pragma unroll
      for (int w = 4; w; w >>= 1)
#pragma unroll
        for (int i = 0; i < w; ++i) ls8[i] += ls8[i + w];
      l = fmaf(l, alpha, ls8[0]);
      if (j > 0 && __any_sync(0xffffffffu, resc)) {
        const int pj = j - 1;
        if (!__all_sync(0xffffffffu, mbar_wait(bar(F_PFREE + (pj & 1)), (pj >> 1) & 1, abort_flag, p.status, detail))) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          float o[32];
          tmem_ld32(tl + 256 + c * 32, reinterpret_cast<uint32_t *>(o));
          tmem_wait_ld();
#pragma unroll
          for (int q = 0; q < 32; ++q) o[q] *= alpha;
          tmem_st32(tl + 256 + c * 32, reinterpret_cast<uint32_t *>(o));
        }
      }
      tmem_st32(tl + sb * 128, pk);
      tmem_st32(tl + sb * 128 + 32, pk + 32);
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(bar(F_PFULL + sb));
    }
    // ---- epilogue
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar(F_OFINAL), 0, abort_flag, p.status, detail));
    tc_fence_after();
    if (ok) {
      float o[D];
#pragma unroll
      for (int c = 0; c < D / 32; ++c) tmem_ld32(tl + 256 + c * 32, reinterpret_cast<uint32_t *>(o + c * 32));
      tmem_wait_ld();
      if (p.num_splits == 1) {
        const float inv = l > 0.f ? 1.f / l : 0.f;
        __nv_bfloat16 *dst = p.out + (((size_t)b * p.max_inline + tok) * p.Hq + hk * p.G + g) * D;
        if (valid) {
#pragma unroll
          for (int q = 0; q < D; ++q) o[q] *= inv;
#pragma unroll
          for (int q = 0; q < D / 8; ++q) st_global16(dst + q * 8, pack8(o + q * 8));
        }
        if (valid && p.lse)
          p.lse[((size_t)b * p.max_inline + tok) * p.Hq + hk * p.G + g] =
              l > 0.f ? (m_used + __log2f(l)) * 0.69314718055994531f : -INFINITY;
      } else {
        float *dst = p.part_o + (part_row0 + row) * D;
        if (valid) {
#pragma unroll
          for (int q = 0; q < D / 4; ++q)
            reinterpret_cast<float4 *>(dst)[q] =
                make_float4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
        }
        p.part_ml[(part_row0 + row) * 2] = (l > 0.f) ? m_used : -INFINITY;
        p.part_ml[(part_row0 + row) * 2 + 1] = l;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if (*abort_flag && lane == 0) mbar_wait(bar(F_OFINAL), 0, abort_flag, p.status, detail);
    __syncwarp();
    tmem_dealloc(tbase, kTmemCols);
  }
}

}  // namespace fused

// Merge the split partials (O unnormalised, m in log2 units, l) of every
// query row by log-sum-exp, lanes over the d columns.  A warp takes R rows
// of one query tile and issues the (m, l) pairs and the O rows of U splits
// for all R rows before using any of them (R * U = 8 loads of 16 bytes in
// flight per lane), so a row costs one L2/DRAM round trip for up to U splits;
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
  const int valid_rows = tin * p.G - (mt * BM + row0);  // rows of this warp that exist
  if (valid_rows <= 0) return;
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
        const float *src = p.part_o + ((base + sp) * BM + row0 + r) * D + lane * CPL;
        if constexpr (CPL == 4) {
          const float4 x = *reinterpret_cast<const float4 *>(src);
          v[r][u][0] = x.x, v[r][u][1] = x.y, v[r][u][2] = x.z, v[r][u][3] = x.w;
        } else {
          static_assert(CPL == 2, "d = 64 or 128");
          const float2 x = *reinterpret_cast<const float2 *>(src);
          v[r][u][0] = x.x, v[r][u][1] = x.y;
        }
      }
    if (s0 == 0) {
#pragma unroll
      for (int r = 0; r < R; ++r) {
        M[r] = ms[r];
#pragma unroll
        for (int o = 16; o; o >>= 1) M[r] = fmaxf(M[r], __shfl_xor_sync(0xffffffffu, M[r], o));
        w[r] = (ms[r] == -INFINITY) ? 0.f : ex2(ms[r] - M[r]);
        Lsum[r] = w[r] * ls[r];
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
    if (r >= valid_rows) break;
    const int rg = mt * BM + row0 + r;
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
  int G, m_tiles, R_pad, splits;
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
    pl.po_bytes = align256(rows * g->head_dim * 4);
    pl.pml_bytes = align256(rows * 2 * 4);
  } else {
    pl.po_bytes = pl.pml_bytes = 0;
  }
  pl.total = pl.q_bytes + pl.po_bytes + pl.pml_bytes;
  return pl;
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
  pp.part_o = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes) : nullptr;
  pp.part_ml = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes + pl.po_bytes) : nullptr;
  pp.status = status;
  pp.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D));

  dim3 grid(((pl.m_tiles + NQ - 1) / NQ) * pl.splits, Hkv, batch);
  cudaError_t e;
  if (D == 128) {
    const int smem = Layout<128>::kAlloc;
    e = cudaFuncSetAttribute(attn_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill smem attribute");
    e = launch_dependent(attn_kernel<128>, grid, dim3(kThreads), smem, stream, tq, tk, tv, pp);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill launch");
  } else {
    const int smem = Layout<64>::kAlloc;
    e = cudaFuncSetAttribute(attn_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill smem attribute");
    e = launch_dependent(attn_kernel<64>, grid, dim3(kThreads), smem, stream, tq, tk, tv, pp);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill launch");
  }
  if (pl.splits > 1) {
    const long long rows = (long long)batch * Hkv * pl.m_tiles * BM;
    e = D == 128 ? launch_combine<128>(rows, pp, stream) : launch_combine<64>(rows, pp, stream);
    if (e != cudaSuccess) return cuda_fail(e, "merge launch");
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill launch");
  return PIC_OK;
}

extern "C" pic_status_t pic_attend_prefill_fused(
    const pic_geom_t *geom, int32_t layer, int32_t batch, int32_t max_inline, const void *q,
    const void *k_new, const void *v_new, const int32_t *inline_pos, const int32_t *inline_len,
    int32_t max_ctx, const int32_t *block_table, int32_t max_pages, int64_t num_pages,
    void *k_cache, void *v_cache, const void *k_pool, const void *v_pool, int64_t pool_tokens,
    int32_t max_docs, const int64_t *doc_token_start, const int32_t *doc_len,
    const int32_t *req_doc_ids, const int32_t *req_num_docs, const int32_t *doc_offset,
    const int32_t *doc_delta, void *out, float *lse, int32_t num_splits, void *workspace,
    size_t workspace_bytes, pic_stream_t stream) {
  using namespace pic;
  using namespace pic::prefill;
  RopeParams rp;
  Plan pl;
  pic_status_t st = check_common("pic_attend_prefill_fused", geom, layer, batch, max_inline,
                                 max_ctx, num_pages, num_splits, workspace, workspace_bytes, &rp,
                                 &pl);
  if (st != PIC_OK) return st;
  if (max_pages <= 0 || pool_tokens <= 0 || max_docs < 0)
    return fail(PIC_ERR_INVALID_ARG, "pic_attend_prefill_fused: sizes must be positive");
  if (max_docs > fused::kMaxDocs)
    return fail(PIC_ERR_UNSUPPORTED, "pic_attend_prefill_fused: max_docs %d > %d", max_docs,
                fused::kMaxDocs);
  if ((long long)geom->num_layers * pool_tokens >= (long long)INT32_MAX)
    return fail(PIC_ERR_UNSUPPORTED, "pic_attend_prefill_fused: pool has more than 2^31 rows");
  if (!inline_pos || !inline_len || !block_table || !k_cache || !v_cache || !k_pool || !v_pool ||
      !out || (max_docs > 0 && (!doc_token_start || !doc_len || !req_doc_ids || !doc_offset ||
                                !doc_delta)) || !req_num_docs)
    return fail(PIC_ERR_INVALID_ARG, "pic_attend_prefill_fused: NULL tensor");
  if ((reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache) |
       reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
       reinterpret_cast<uintptr_t>(out)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_attend_prefill_fused: bf16 tensors must be 16-byte aligned");
  st = check_projections("pic_attend_prefill_fused", q, k_new, v_new);
  if (st != PIC_OK) return st;
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_attend_prefill_fused: no device status word");
  if (q) {  // the inline tokens' RoPE and append first (slots from the block table)
    st = launch_append("pic_attend_prefill_fused", geom, rp, pl, layer, batch, max_inline, q,
                       k_new, v_new, inline_pos, inline_len, nullptr, block_table, max_pages,
                       max_ctx, num_pages, k_cache, v_cache, workspace, stream);
    if (st != PIC_OK) return st;
  }
  const int D = geom->head_dim, Hkv = geom->num_kv_heads;
  const long long rows_total = (long long)geom->num_layers * num_pages * Hkv * 16;
  uint8_t *ws = static_cast<uint8_t *>(workspace);

  CUtensorMap tq, tk, tv, tkp, tvp;
  st = encode_tmap_2d(&tq, ws, D, (uint64_t)batch * Hkv * pl.R_pad, (uint64_t)D * 2, 64, BM);
  if (st == PIC_OK) st = encode_tmap_2d(&tk, k_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
  if (st == PIC_OK) st = encode_tmap_2d(&tv, v_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
  const uint64_t pool_rows = (uint64_t)geom->num_layers * pool_tokens;
  if (st == PIC_OK)
    st = encode_tmap_3d(&tkp, k_pool, D, Hkv, pool_rows, (uint64_t)D * 2, (uint64_t)Hkv * D * 2,
                        64, 1, fused::BN);
  if (st == PIC_OK)
    st = encode_tmap_3d(&tvp, v_pool, D, Hkv, pool_rows, (uint64_t)D * 2, (uint64_t)Hkv * D * 2,
                        64, 1, fused::BN);
  if (st != PIC_OK) return st;

  fused::FParams fp;
  Params &pp = fp.base;
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
  pp.part_o = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes) : nullptr;
  pp.part_ml = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes + pl.po_bytes) : nullptr;
  pp.status = status;
  pp.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D));
  fp.rp = rp;
  fp.pool_tokens = pool_tokens;
  fp.max_docs = max_docs;
  fp.layer = layer;
  fp.num_docs = req_num_docs;
  fp.doc_offset = doc_offset;
  fp.doc_delta = doc_delta;
  fp.ids = req_doc_ids;
  fp.doc_len = doc_len;
  fp.doc_start = doc_token_start;

  dim3 grid(pl.m_tiles * pl.splits, Hkv, batch);
  cudaError_t e;
  if (D == 128) {
    const int smem = fused::Layout<128>::kAlloc;
    e = cudaFuncSetAttribute(fused::attn_fused_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill_fused smem attribute");
    e = launch_dependent(fused::attn_fused_kernel<128>, grid, dim3(fused::kThreads), smem, stream,
                         tq, tk, tv, tkp, tvp, fp);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill_fused launch");
  } else {
    const int smem = fused::Layout<64>::kAlloc;
    e = cudaFuncSetAttribute(fused::attn_fused_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill_fused smem attribute");
    e = launch_dependent(fused::attn_fused_kernel<64>, grid, dim3(fused::kThreads), smem, stream,
                         tq, tk, tv, tkp, tvp, fp);
    if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill_fused launch");
  }
  if (pl.splits > 1) {
    const long long crows = (long long)batch * Hkv * pl.m_tiles * BM;
    e = D == 128 ? launch_combine<128>(crows, pp, stream) : launch_combine<64>(crows, pp, stream);
    if (e != cudaSuccess) return cuda_fail(e, "merge launch");
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_attend_prefill_fused launch");
  return PIC_OK;
}
