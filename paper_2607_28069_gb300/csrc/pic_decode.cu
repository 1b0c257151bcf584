// pic_attend_decode: one step of plain autoregressive decoding over the
// completed stitched cache (appendix "Position-Independent Linking": after the
// first token, generation proceeds as usual on the linked cache).
//
// Decode reads every cached key and value of the request once per step and
// does 2*G*d multiply-adds per key: HBM-bound.  Launches per call (one layer):
//  1. decode_append_kernel: R(pos) k_new and v_new into slot(pos); the query
//     rotated at pos into a bf16 workspace.
//  2. decode_attn_kernel: one CTA per (key split, kv head, request), four
//     warps, each warp an independent stream over the split's pages (page
//     w, w+4, ...).  Lane 0 of each warp keeps a 3-deep ring of TMA loads
//     (one 16-key K page and V page, 128-byte swizzled so the ldmatrix reads
//     below are bank-conflict free).  Scores S^T = K q^T come from
//     m16n8k16 warp MMAs with the page's 16 keys as M and up to 8 query heads
//     of the GQA group as N; P^T is turned into the B operand of the
//     O^T += V^T P^T MMA in registers with movmatrix.  The four warps' states
//     are merged through shared memory at the end.
//  3. decode_combine_kernel (only with several splits): log-sum-exp merge.
#include <algorithm>
#include <mutex>

#include "pic_internal.cuh"

namespace pic {
namespace decode {

constexpr int kWarps = 4;
constexpr int kThreads = 32 * kWarps;
constexpr int NSTG = 3;
constexpr int kMaxSplits = 64;

template <int D>
struct Layout {
  static constexpr int kPage = 16 * D * 2;        // one K (or V) page of one head
  static constexpr int kStage = 2 * kPage;        // K + V
  static constexpr int kWarpBytes = NSTG * kStage;
  static constexpr int kBar = kWarps * kWarpBytes;
  static constexpr int kBytes = kBar + kWarps * NSTG * 8 + 16;
  static constexpr int kAlloc = kBytes + 1024;
};

struct Params {
  int Hq, Hkv, G, max_pages, splits, pages_per_split, pos_offset;
  long long num_pages, layer_row0;
  const int32_t *pos, *block_table;
  const __nv_bfloat16 *qrot;  // [B][Hq][D]
  __nv_bfloat16 *out;
  float *lse, *part_o, *part_ml;
  int32_t *status;
  float scale_log2;
};

template <int D, int NT>
__global__ void __launch_bounds__(kThreads)
    decode_attn_kernel(const __grid_constant__ CUtensorMap tm_k,
                       const __grid_constant__ CUtensorMap tm_v, Params p) {
  using L = Layout<D>;
  constexpr int PANELS = D / 64;
  constexpr int KS = D / 16;  // k-steps over d
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~(uintptr_t)1023);
  const uint32_t sbase = smem_u32(smem);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + L::kBar + kWarps * NSTG * 8);

  const int split = blockIdx.x, hk = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tig = lane & 3;

  // set-up that reads nothing another kernel writes, then wait for the
  // kernel before (programmatic dependent launch)
  if (threadIdx.x == 0) {
    for (int i = 0; i < kWarps * NSTG; ++i) mbar_init(sbase + L::kBar + 8 * i, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (lane == 0) {
    prefetch_tmap(&tm_k);
    prefetch_tmap(&tm_v);
  }
  __syncthreads();
  asm volatile("griddepcontrol.wait;" ::: "memory");

  const int pos = p.pos[b] + p.pos_offset;
  const int npages = pos >= 0 ? pos / 16 + 1 : 0;
  // max_ctx sized the split plan: keys past the last split's pages would be
  // left out, so that is a device-checked error (the step's output for the
  // request is then incomplete)
  if (split == p.splits - 1 && threadIdx.x == 0 && npages > p.splits * p.pages_per_split)
    dev_fail(p.status, PIC_DEV_CTX_OVERFLOW, b);
  const int pg_begin = split * p.pages_per_split;
  const int pg_end = min(npages, pg_begin + p.pages_per_split);
  const int32_t *bt = p.block_table + (size_t)b * p.max_pages;

  const uint32_t wbase = sbase + warp * L::kWarpBytes;
  auto full = [&](int s) { return sbase + L::kBar + 8u * (uint32_t)(warp * NSTG + s); };
  // pages of this warp: pg_begin + warp + 4 i
  const int my_first = pg_begin + warp;
  const int cw = my_first < pg_end ? (pg_end - my_first + kWarps - 1) / kWarps : 0;

  auto issue = [&](int i) {  // lane 0 only
    const int pidx = my_first + kWarps * i;
    int y = -1;
    if (pidx < p.max_pages) {
      const int page = bt[pidx];
      if (page >= 0 && page < p.num_pages) y = (int)(p.layer_row0 + ((long long)page * p.Hkv + hk) * 16);
      else dev_fail(p.status, PIC_DEV_BAD_PAGE, b);
    } else {
      dev_fail(p.status, PIC_DEV_BLOCK_TABLE_SHORT, b);
    }
    if (y < 0) y = 0x7fffff00;  // out of the tensor: TMA fills zeros
    const int s = i % NSTG;
    const uint32_t dst = wbase + s * L::kStage;
    mbar_expect_tx(full(s), L::kStage);
    for (int pn = 0; pn < PANELS; ++pn) {
      tma_load_2d(dst + pn * 2048, &tm_k, pn * 64, y, full(s));
      tma_load_2d(dst + L::kPage + pn * 2048, &tm_v, pn * 64, y, full(s));
    }
  };
  if (lane == 0)
    for (int i = 0; i < min(cw, NSTG); ++i) issue(i);

  // query fragments (B operand of S^T = K q^T): heads nt*8 + gid of the group
  uint32_t qb[NT][KS][2];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    const int hh = nt * 8 + gid;
    const bool hv = hh < p.G;
    const uint32_t *qr = reinterpret_cast<const uint32_t *>(
        p.qrot + ((size_t)b * p.Hq + hk * p.G + (hv ? hh : 0)) * D);
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
      qb[nt][kk][0] = hv ? qr[(kk * 16 + 2 * tig) / 2] : 0u;
      qb[nt][kk][1] = hv ? qr[(kk * 16 + 8 + 2 * tig) / 2] : 0u;
    }
  }

  float m[NT][2], l[NT][2], o[NT][KS][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
    for (int j = 0; j < 2; ++j) { m[nt][j] = -INFINITY; l[nt][j] = 0.f; }
#pragma unroll
    for (int mt = 0; mt < KS; ++mt)
#pragma unroll
      for (int q = 0; q < 4; ++q) o[nt][mt][q] = 0.f;
  }

  int done = 0;
  for (int i = 0; i < cw; ++i) {
    const int s = i % NSTG;
    const bool ok = mbar_wait(full(s), (i / NSTG) & 1, abort_flag, p.status, b);
    if (!__all_sync(0xffffffffu, ok)) break;
    done = i + 1;
    const uint32_t ks = wbase + s * L::kStage, vs = ks + L::kPage;
    const int key0 = (my_first + kWarps * i) * 16;
    // ---- S^T[16 keys][8 heads] per n-tile
    float sacc[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int q = 0; q < 4; ++q) sacc[nt][q] = 0.f;
    {
      const int mi = lane >> 3, rr = (mi & 1) * 8 + (lane & 7);
#pragma unroll
      for (int kk = 0; kk < KS; ++kk) {
        const int col = kk * 16 + (mi >> 1) * 8;
        uint32_t a[4];
        ldsm_x4(ks + (col >> 6) * 2048 + sw128_offset(rr, col & 63), a);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma16816(sacc[nt], a, qb[nt][kk][0], qb[nt][kk][1]);
      }
    }
    // ---- online softmax (thread: keys gid, gid+8; heads 2tig, 2tig+1 of each n-tile)
    const bool m0 = key0 + gid > pos, m1 = key0 + gid + 8 > pos;
    uint32_t pb[NT][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      float pv[2][2];
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        const float s0 = m0 ? -INFINITY : sacc[nt][j] * p.scale_log2;
        const float s1 = m1 ? -INFINITY : sacc[nt][2 + j] * p.scale_log2;
        float mx = fmaxf(s0, s1);
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
        mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
        const float mn = fmaxf(m[nt][j], mx);
        const float mref = mn == -INFINITY ? 0.f : mn;
        const float alpha = ex2(m[nt][j] - mref);
        m[nt][j] = mn;
        pv[0][j] = ex2(s0 - mref);
        pv[1][j] = ex2(s1 - mref);
        l[nt][j] = l[nt][j] * alpha + pv[0][j] + pv[1][j];
#pragma unroll
        for (int mt = 0; mt < KS; ++mt) {
          o[nt][mt][j] *= alpha;
          o[nt][mt][2 + j] *= alpha;
        }
      }
      pb[nt][0] = movm_t(pack2(pv[0][0], pv[0][1]));
      pb[nt][1] = movm_t(pack2(pv[1][0], pv[1][1]));
    }
    // ---- O^T[d][heads] += V^T P^T
    {
      const int mi = lane >> 3, rr = (mi >> 1) * 8 + (lane & 7);
#pragma unroll
      for (int mt = 0; mt < KS; ++mt) {
        const int col = mt * 16 + (mi & 1) * 8;
        uint32_t a[4];
        ldsm_x4_t(vs + (col >> 6) * 2048 + sw128_offset(rr, col & 63), a);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma16816(o[nt][mt], a, pb[nt][0], pb[nt][1]);
      }
    }
    __syncwarp();
    if (lane == 0 && i + NSTG < cw) issue(i + NSTG);
  }

  if (done < cw) {
    // aborted: let the loads already issued land before the ring is reused
    for (int i = done; i < min(cw, done + NSTG); ++i)
      mbar_wait(full(i % NSTG), (i / NSTG) & 1, abort_flag, p.status, b);
  }
  // ---- reduce l over the 8 key lanes, then merge the four warps
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      float v = l[nt][j];
      v += __shfl_xor_sync(0xffffffffu, v, 4);
      v += __shfl_xor_sync(0xffffffffu, v, 8);
      v += __shfl_xor_sync(0xffffffffu, v, 16);
      l[nt][j] = v;
    }
  __syncthreads();  // every warp finished with its ring: reuse it for the merge
  constexpr int HMAX = NT * 8;
  float *so = reinterpret_cast<float *>(smem);                  // [warps][HMAX][D]
  float *sm = so + kWarps * HMAX * D;                            // [warps][HMAX]
  float *sl = sm + kWarps * HMAX;                                // [warps][HMAX]
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int hh = nt * 8 + 2 * tig + j;
      if (gid == 0) {
        sm[warp * HMAX + hh] = m[nt][j];
        sl[warp * HMAX + hh] = l[nt][j];
      }
#pragma unroll
      for (int mt = 0; mt < KS; ++mt) {
        so[(warp * HMAX + hh) * D + mt * 16 + gid] = o[nt][mt][j];
        so[(warp * HMAX + hh) * D + mt * 16 + gid + 8] = o[nt][mt][2 + j];
      }
    }
  __syncthreads();
  const bool single = p.splits == 1;
  for (int e = threadIdx.x; e < p.G * D; e += kThreads) {
    const int hh = e / D, d = e % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) M = fmaxf(M, sm[w * HMAX + hh]);
    float acc = 0.f, Ls = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
      const float mw = sm[w * HMAX + hh];
      const float wt = mw == -INFINITY ? 0.f : ex2(mw - M);
      acc = fmaf(wt, so[(w * HMAX + hh) * D + d], acc);
      Ls = fmaf(wt, sl[w * HMAX + hh], Ls);
    }
    const size_t h = (size_t)b * p.Hq + hk * p.G + hh;
    if (single) {
      p.out[h * D + d] = __float2bfloat16_rn(Ls > 0.f ? acc / Ls : 0.f);
      if (d == 0 && p.lse) p.lse[h] = Ls > 0.f ? (M + __log2f(Ls)) * 0.69314718055994531f : -INFINITY;
    } else {
      p.part_o[(h * p.splits + split) * D + d] = acc;
      if (d == 0) {
        p.part_ml[(h * p.splits + split) * 2] = Ls > 0.f ? M : -INFINITY;
        p.part_ml[(h * p.splits + split) * 2 + 1] = Ls;
      }
    }
  }
  // release the dependent launch (merge, or the next layer's append) last
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Merge of the split partials of one (request, query head) row by
// log-sum-exp: o = sum_s w_s O_s / sum_s w_s l_s with w_s = 2^(m_s - M).
// Lane s holds split s's (m, l) (and lane s - 32 split s >= 32), so the
// maximum and the weight sum are warp reductions, and the O rows of eight
// splits are loaded before any is used (the first sixteen together with
// the (m, l) pairs): a row costs a few L2 round trips however many splits
// it has, not one per split.
template <int D>
__global__ void decode_combine_kernel(Params p) {
  static_assert(kMaxSplits <= 64, "two (m, l) slots per lane");
  constexpr int CPL = D / 32, U = 8;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int h = blockIdx.x, b = blockIdx.y, lane = threadIdx.x;
  const size_t hrow = (size_t)b * p.Hq + h;
  const int S = p.splits;
  // the first sixteen splits' O rows go out with the (m, l) loads
  const float *src = p.part_o + hrow * S * D + lane;
  float v0[U][CPL], v1[U][CPL];
#pragma unroll
  for (int u = 0; u < U; ++u)
#pragma unroll
    for (int q = 0; q < CPL; ++q) {
      v0[u][q] = u < S ? src[(size_t)u * D + q * 32] : 0.f;
      v1[u][q] = U + u < S ? src[(size_t)(U + u) * D + q * 32] : 0.f;
    }
  float mA = -INFINITY, lA = 0.f, mB = -INFINITY, lB = 0.f;
  if (lane < S) {
    const float2 ml = *reinterpret_cast<const float2 *>(p.part_ml + (hrow * S + lane) * 2);
    mA = ml.x, lA = ml.y;
  }
  if (lane + 32 < S) {
    const float2 ml = *reinterpret_cast<const float2 *>(p.part_ml + (hrow * S + lane + 32) * 2);
    mB = ml.x, lB = ml.y;
  }
  float M = fmaxf(mA, mB);
#pragma unroll
  for (int o = 16; o; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
  const float wA = mA == -INFINITY ? 0.f : ex2(mA - M);
  const float wB = mB == -INFINITY ? 0.f : ex2(mB - M);
  float Ls = fmaf(wA, lA, wB * lB);
#pragma unroll
  for (int o = 16; o; o >>= 1) Ls += __shfl_xor_sync(0xffffffffu, Ls, o);
  float acc[CPL];
#pragma unroll
  for (int q = 0; q < CPL; ++q) acc[q] = 0.f;
  for (int s0 = 0; s0 < S; s0 += U) {
    float v[U][CPL];
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int q = 0; q < CPL; ++q)
        v[u][q] = s0 == 0   ? v0[u][q]
                  : s0 == U ? v1[u][q]
                            : (s0 + u < S ? src[(size_t)(s0 + u) * D + q * 32] : 0.f);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int sp = s0 + u;
      if (sp >= S) break;
      const float w = __shfl_sync(0xffffffffu, sp < 32 ? wA : wB, sp & 31);
      if (w == 0.f) continue;  // an empty split; its rows were never written
#pragma unroll
      for (int q = 0; q < CPL; ++q) acc[q] = fmaf(w, v[u][q], acc[q]);
    }
  }
  const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
#pragma unroll
  for (int q = 0; q < CPL; ++q) p.out[hrow * D + q * 32 + lane] = __float2bfloat16_rn(acc[q] * inv);
  if (lane == 0 && p.lse) p.lse[hrow] = Ls > 0.f ? (M + __log2f(Ls)) * 0.69314718055994531f : -INFINITY;
}

struct AppendArgs {
  int Hq, Hkv, max_pages, pos_offset, layer;
  long long num_pages;
  const __nv_bfloat16 *q, *k, *v;
  const int32_t *pos, *block_table;
  __nv_bfloat16 *k_cache, *v_cache, *qrot;  // cache pointers at the layer
  int32_t *status;
};

template <int D>
__global__ void __launch_bounds__(128) decode_append_kernel(AppendArgs a, RopeParams rp) {
  constexpr int HALF = D / 2, KC = D / 16, VC = D / 8;
  constexpr int R = 2;  // chunks per thread whose loads go out before the position is known
  pdl_entry();
  const int b = blockIdx.x, tid = threadIdx.x;
  __shared__ float2 cs[HALF];
  const int nK = a.Hkv * KC, nV = a.Hkv * VC, nQ = a.Hq * KC;
  // the token's projections do not depend on its position: their first
  // chunks are loaded before it is (the rest, if any, after)
  uint4 ka[R], kb[R], vv[R], qa[R], qb[R];
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int e = tid + (int)blockDim.x * i;
    if (e < nK) {
      const PairChunk pc = pair_chunk(e % KC, HALF, rp.style);
      const __nv_bfloat16 *src = a.k + ((size_t)b * a.Hkv + e / KC) * D;
      ka[i] = ld_stream(src + pc.off_a);
      kb[i] = ld_stream(src + pc.off_b);
    }
    if (e < nV) vv[i] = ld_stream(a.v + ((size_t)b * a.Hkv + e / VC) * D + (e % VC) * 8);
    if (e < nQ) {
      const PairChunk pc = pair_chunk(e % KC, HALF, rp.style);
      const __nv_bfloat16 *src = a.q + ((size_t)b * a.Hq + e / KC) * D;
      qa[i] = ld_stream(src + pc.off_a);
      qb[i] = ld_stream(src + pc.off_b);
    }
  }
  const int pos = a.pos[b] + a.pos_offset;
  long long page = -1;
  if (pos < 0 || pos / 16 >= a.max_pages) {
    if (tid == 0) dev_fail(a.status, PIC_DEV_BAD_POSITION, b);
  } else {
    page = a.block_table[(size_t)b * a.max_pages + pos / 16];
    if (page < 0 || page >= a.num_pages) {
      if (tid == 0) dev_fail(a.status, PIC_DEV_BAD_PAGE, b);
      page = -1;
    }
  }
  for (int i = tid; i < HALF; i += blockDim.x)
    cs[i] = rope_cos_sin(pos > 0 ? pos : 0, rope_theta(rp, a.layer, i));
  __syncthreads();
  const int r = pos & 15;
  auto k_dst = [&](int e) { return a.k_cache + ((page * a.Hkv + e / KC) * 16 + r) * D; };
  auto v_dst = [&](int e) { return a.v_cache + ((page * a.Hkv + e / VC) * 16 + r) * D + (e % VC) * 8; };
  auto q_dst = [&](int e) { return a.qrot + ((size_t)b * a.Hq + e / KC) * D; };
  if (page >= 0) {
#pragma unroll
    for (int i = 0; i < R; ++i) {
      const int e = tid + (int)blockDim.x * i;
      if (e < nK) rotate_store(ka[i], kb[i], k_dst(e), pair_chunk(e % KC, HALF, rp.style), rp.style, cs + 8 * (e % KC));
      if (e < nV) st_global16(v_dst(e), vv[i]);
    }
    for (int e = tid + (int)blockDim.x * R; e < nK; e += blockDim.x)
      rotate_chunk(a.k + ((size_t)b * a.Hkv + e / KC) * D, k_dst(e), e % KC, HALF, rp.style,
                   cs + 8 * (e % KC), true);
    for (int e = tid + (int)blockDim.x * R; e < nV; e += blockDim.x)
      st_global16(v_dst(e), ld_stream(a.v + ((size_t)b * a.Hkv + e / VC) * D + (e % VC) * 8));
  }
#pragma unroll
  for (int i = 0; i < R; ++i) {
    const int e = tid + (int)blockDim.x * i;
    if (e < nQ) rotate_store(qa[i], qb[i], q_dst(e), pair_chunk(e % KC, HALF, rp.style), rp.style, cs + 8 * (e % KC));
  }
  for (int e = tid + (int)blockDim.x * R; e < nQ; e += blockDim.x)
    rotate_chunk(a.q + ((size_t)b * a.Hq + e / KC) * D, q_dst(e), e % KC, HALF, rp.style,
                 cs + 8 * (e % KC), true);
}

struct Plan {
  int splits, pages_per_split;
  size_t q_bytes, po_bytes, pml_bytes, total;
};

inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

inline Plan plan(const pic_geom_t *g, int batch, int max_ctx, int num_splits) {
  Plan pl;
  const int pages = (max_ctx + 15) / 16;
  if (num_splits <= 0) {
    const long long units = (long long)batch * g->num_kv_heads;
    int s = (int)((8LL * 152 + units - 1) / units);
    s = std::min(s, std::max(1, pages / 16));  // at least ~4 pages per warp
    num_splits = std::max(1, std::min(s, kMaxSplits));
  }
  num_splits = std::min(num_splits, pages);
  pl.splits = std::max(1, num_splits);
  pl.pages_per_split = (pages + pl.splits - 1) / pl.splits;
  pl.q_bytes = align256((size_t)batch * g->num_q_heads * g->head_dim * 2);
  if (pl.splits > 1) {
    pl.po_bytes = align256((size_t)batch * g->num_q_heads * pl.splits * g->head_dim * 4);
    pl.pml_bytes = align256((size_t)batch * g->num_q_heads * pl.splits * 2 * 4);
  } else {
    pl.po_bytes = pl.pml_bytes = 0;
  }
  pl.total = pl.q_bytes + pl.po_bytes + pl.pml_bytes;
  return pl;
}

template <int D, int NT>
cudaError_t launch_attn(dim3 grid, cudaStream_t stream, const CUtensorMap &tk,
                        const CUtensorMap &tv, const Params &pp) {
  const int smem = Layout<D>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(decode_attn_kernel<D, NT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = launch_dependent(decode_attn_kernel<D, NT>, grid, dim3(kThreads), smem, stream, tk, tv, pp);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace decode
}  // namespace pic

extern "C" size_t pic_decode_workspace_size(const pic_geom_t *geom, int32_t batch, int32_t max_ctx,
                                            int32_t num_splits) {
  if (!geom || batch <= 0 || max_ctx <= 0 || geom->num_kv_heads <= 0) return 0;
  return pic::decode::plan(geom, batch, max_ctx, num_splits).total;
}

extern "C" int32_t pic_decode_num_splits(const pic_geom_t *geom, int32_t batch, int32_t max_ctx,
                                         int32_t num_splits) {
  if (!geom || batch <= 0 || max_ctx <= 0 || geom->num_kv_heads <= 0 || num_splits < 0 ||
      num_splits > pic::decode::kMaxSplits)
    return 0;
  return pic::decode::plan(geom, batch, max_ctx, num_splits).splits;
}

namespace pic {
namespace decode {

// Host checks shared by pic_attend_decode and pic_attend_decode_noalloc
// (everything but the scratch); fills the rotary parameters.
static pic_status_t check_step(const char *who, const pic_geom_t *geom, RopeParams *rp,
                               int32_t layer, int32_t batch, const void *q, const void *k_new,
                               const void *v_new, const int32_t *pos, const int32_t *block_table,
                               int32_t max_pages, int64_t num_pages, const void *k_cache,
                               const void *v_cache, const void *out, int32_t max_ctx,
                               int32_t num_splits) {
  pic_status_t st = make_rope(geom, rp);
  if (st != PIC_OK) return st;
  if (layer < 0 || layer >= geom->num_layers)
    return fail(PIC_ERR_INVALID_ARG, "%s: layer %d outside [0, %d)", who, layer,
                geom->num_layers);
  if (batch <= 0 || max_pages <= 0 || num_pages <= 0 || max_ctx <= 0)
    return fail(PIC_ERR_INVALID_ARG, "%s: sizes must be positive", who);
  if (num_splits < 0 || num_splits > kMaxSplits)
    return fail(PIC_ERR_INVALID_ARG, "%s: num_splits %d outside [0, %d]", who, num_splits,
                kMaxSplits);
  if (geom->num_q_heads / geom->num_kv_heads > 16)
    return fail(PIC_ERR_UNSUPPORTED, "%s: more than 16 query heads per kv head", who);
  if (!q || !k_new || !v_new || !pos || !block_table || !k_cache || !v_cache || !out)
    return fail(PIC_ERR_INVALID_ARG, "%s: NULL tensor", who);
  if ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k_new) |
       reinterpret_cast<uintptr_t>(v_new) | reinterpret_cast<uintptr_t>(k_cache) |
       reinterpret_cast<uintptr_t>(v_cache)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "%s: bf16 tensors must be 16-byte aligned", who);
  const long long rows_total =
      (long long)geom->num_layers * num_pages * geom->num_kv_heads * 16;
  if (rows_total + 16 >= 0x7fffff00LL)
    return fail(PIC_ERR_UNSUPPORTED, "%s: cache has more than 2^31 rows", who);
  if (batch > 65535 || geom->num_kv_heads > 65535)
    return fail(PIC_ERR_UNSUPPORTED, "%s: grid too large", who);
  return PIC_OK;
}

// The launches of one decoding step of one layer (append, attention, merge
// when split) with the scratch at `ws` laid out by `pl`.
static pic_status_t launch_step(const char *who, const pic_geom_t *geom, const RopeParams &rp,
                                int32_t layer, int32_t batch, const void *q, const void *k_new,
                                const void *v_new, const int32_t *pos, int32_t pos_offset,
                                const int32_t *block_table, int32_t max_pages, int64_t num_pages,
                                void *k_cache, void *v_cache, void *out, float *lse,
                                const Plan &pl, uint8_t *ws, pic_stream_t stream) {
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "%s: no device status word", who);
  const int D = geom->head_dim, Hkv = geom->num_kv_heads;
  const int G = geom->num_q_heads / Hkv;
  const long long rows_total = (long long)geom->num_layers * num_pages * Hkv * 16;
  const size_t layer_elems = (size_t)num_pages * Hkv * 16 * D;

  AppendArgs aa;
  aa.Hq = geom->num_q_heads;
  aa.Hkv = Hkv;
  aa.max_pages = max_pages;
  aa.pos_offset = pos_offset;
  aa.layer = layer;
  aa.num_pages = num_pages;
  aa.q = static_cast<const __nv_bfloat16 *>(q);
  aa.k = static_cast<const __nv_bfloat16 *>(k_new);
  aa.v = static_cast<const __nv_bfloat16 *>(v_new);
  aa.pos = pos;
  aa.block_table = block_table;
  aa.k_cache = static_cast<__nv_bfloat16 *>(k_cache) + (size_t)layer * layer_elems;
  aa.v_cache = static_cast<__nv_bfloat16 *>(v_cache) + (size_t)layer * layer_elems;
  aa.qrot = reinterpret_cast<__nv_bfloat16 *>(ws);
  aa.status = status;
  {
    const cudaError_t ae =
        D == 128 ? launch_dependent(decode_append_kernel<128>, dim3(batch), dim3(128), 0, stream, aa, rp)
                 : launch_dependent(decode_append_kernel<64>, dim3(batch), dim3(128), 0, stream, aa, rp);
    if (ae != cudaSuccess) return cuda_fail(ae, "decode append launch");
  }

  CUtensorMap tk, tv;
  pic_status_t st = encode_tmap_2d(&tk, k_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
  if (st == PIC_OK) st = encode_tmap_2d(&tv, v_cache, D, rows_total, (uint64_t)D * 2, 64, 16);
  if (st != PIC_OK) return st;

  Params pp;
  pp.Hq = geom->num_q_heads;
  pp.Hkv = Hkv;
  pp.G = G;
  pp.max_pages = max_pages;
  pp.splits = pl.splits;
  pp.pages_per_split = pl.pages_per_split;
  pp.pos_offset = pos_offset;
  pp.num_pages = num_pages;
  pp.layer_row0 = (long long)layer * num_pages * Hkv * 16;
  pp.pos = pos;
  pp.block_table = block_table;
  pp.qrot = aa.qrot;
  pp.out = static_cast<__nv_bfloat16 *>(out);
  pp.lse = lse;
  pp.part_o = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes) : nullptr;
  pp.part_ml = pl.splits > 1 ? reinterpret_cast<float *>(ws + pl.q_bytes + pl.po_bytes) : nullptr;
  pp.status = status;
  pp.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)D));

  dim3 grid(pl.splits, Hkv, batch);
  cudaError_t e;
  if (D == 128) e = G <= 8 ? launch_attn<128, 1>(grid, stream, tk, tv, pp) : launch_attn<128, 2>(grid, stream, tk, tv, pp);
  else e = G <= 8 ? launch_attn<64, 1>(grid, stream, tk, tv, pp) : launch_attn<64, 2>(grid, stream, tk, tv, pp);
  if (e != cudaSuccess) return cuda_fail(e, "decode attention launch");
  if (pl.splits > 1) {
    dim3 cgrid(geom->num_q_heads, batch);
    const cudaError_t ce =
        D == 128 ? launch_dependent(decode_combine_kernel<128>, cgrid, dim3(32), 0, stream, pp)
                 : launch_dependent(decode_combine_kernel<64>, cgrid, dim3(32), 0, stream, pp);
    if (ce != cudaSuccess) return cuda_fail(ce, "decode merge launch");
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "decode launch");
  return PIC_OK;
}

}  // namespace decode
}  // namespace pic

extern "C" pic_status_t pic_attend_decode(const pic_geom_t *geom, int32_t layer, int32_t batch,
                                          const void *q, const void *k_new, const void *v_new,
                                          const int32_t *pos, int32_t pos_offset,
                                          const int32_t *block_table,
                                          int32_t max_pages, int64_t num_pages, void *k_cache,
                                          void *v_cache, void *out, float *lse, int32_t max_ctx,
                                          int32_t num_splits, void *workspace,
                                          size_t workspace_bytes, pic_stream_t stream) {
  using namespace pic;
  using namespace pic::decode;
  static const char *who = "pic_attend_decode";
  RopeParams rp;
  pic_status_t st = check_step(who, geom, &rp, layer, batch, q, k_new, v_new, pos, block_table,
                               max_pages, num_pages, k_cache, v_cache, out, max_ctx, num_splits);
  if (st != PIC_OK) return st;
  const Plan pl = plan(geom, batch, max_ctx, num_splits);
  if (!workspace || workspace_bytes < pl.total || (reinterpret_cast<uintptr_t>(workspace) & 255))
    return fail(PIC_ERR_WORKSPACE, "pic_attend_decode: workspace needs %zu bytes, 256-aligned",
                pl.total);
  return launch_step(who, geom, rp, layer, batch, q, k_new, v_new, pos, pos_offset, block_table,
                     max_pages, num_pages, k_cache, v_cache, out, lse, pl,
                     static_cast<uint8_t *>(workspace), stream);
}

// ---------------------------------------------------------------------------
// pic_attend_decode_noalloc: the same decoding step for callers that cannot
// allocate device memory on the step path.
//
// Some callers cannot call cudaMalloc (or any allocator) while they decode: an
// engine that has handed its whole memory budget to the KV cache, a runtime
// that forbids allocation after start-up, or an embedding that only owns the
// tensors it passes in.  For them this entry point takes no workspace: its
// scratch (the rotated queries and the per-split partial softmax states) lives
// in the file-scope device array below, which every GPU that loads the library
// holds until the process exits.
//
// Set-up: the first call on each device (with that device current) looks up
// the array's device address with cudaGetSymbolAddress and caches it, per
// device context (a device reset replaces the context, and the address is
// looked up again); make that first call before any stream capture.  The array is shared by every
// call on the device and keeps the last call's contents: calls that overlap on
// the GPU (for example on two streams) race on it.  Nothing in it needs to
// start at zero: each call writes every scratch value before reading it.
namespace pic {
namespace decode {

constexpr size_t kNoAllocScratchBytes = 8u << 20;  // 8 MiB per device
static __device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocScratchBytes];

static uint8_t *noalloc_scratch_ptr(pic_status_t *st) {
  constexpr int kMaxDev = 64;
  static uint8_t *ptrs[kMaxDev] = {nullptr};
  static unsigned long long ctx_ids[kMaxDev] = {0};
  static std::mutex mu;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDev) {
    *st = e != cudaSuccess ? cuda_fail(e, "pic_attend_decode_noalloc: cudaGetDevice")
                           : fail(PIC_ERR_CUDA, "pic_attend_decode_noalloc: device %d", dev);
    return nullptr;
  }
  std::lock_guard<std::mutex> lk(mu);
  // Set-up once per device (per device context: after a device reset the
  // array has a new address in the new context, so it is looked up again).
  const unsigned long long id = current_context_id();
  if (!ptrs[dev] || id == 0 || id != ctx_ids[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) {
      *st = cuda_fail(e, "pic_attend_decode_noalloc: cudaGetSymbolAddress");
      return nullptr;
    }
    ptrs[dev] = static_cast<uint8_t *>(p);
    ctx_ids[dev] = current_context_id();
  }
  *st = PIC_OK;
  return ptrs[dev];
}

}  // namespace decode
}  // namespace pic

extern "C" pic_status_t pic_attend_decode_noalloc(const pic_geom_t *geom, int32_t layer,
                                                  int32_t batch, const void *q, const void *k_new,
                                                  const void *v_new, const int32_t *pos,
                                                  int32_t pos_offset, const int32_t *block_table,
                                                  int32_t max_pages, int64_t num_pages,
                                                  void *k_cache, void *v_cache, void *out,
                                                  float *lse, int32_t max_ctx, int32_t num_splits,
                                                  pic_stream_t stream) {
  using namespace pic;
  using namespace pic::decode;
  static const char *who = "pic_attend_decode_noalloc";
  RopeParams rp;
  pic_status_t st = check_step(who, geom, &rp, layer, batch, q, k_new, v_new, pos, block_table,
                               max_pages, num_pages, k_cache, v_cache, out, max_ctx, num_splits);
  if (st != PIC_OK) return st;
  // Scratch must fit the built-in array: the automatic split count is lowered
  // until it does; an explicit split count that does not fit is rejected.
  Plan pl = plan(geom, batch, max_ctx, num_splits);
  if (num_splits == 0)
    while (pl.total > kNoAllocScratchBytes && pl.splits > 1)
      pl = plan(geom, batch, max_ctx, pl.splits - 1);
  if (pl.total > kNoAllocScratchBytes)
    return fail(PIC_ERR_WORKSPACE,
                "pic_attend_decode_noalloc: needs %zu bytes of scratch, the built-in array holds "
                "%zu (fewer splits or a smaller batch may fit; pic_attend_decode takes a "
                "caller workspace instead)",
                pl.total, kNoAllocScratchBytes);
  uint8_t *ws = noalloc_scratch_ptr(&st);
  if (!ws) return st;
  return launch_step(who, geom, rp, layer, batch, q, k_new, v_new, pos, pos_offset, block_table,
                     max_pages, num_pages, k_cache, v_cache, out, lse, pl, ws, stream);
}
