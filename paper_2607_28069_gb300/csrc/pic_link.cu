// pic_link: the link step of a cache hit in one launch -- the logical layout
// and slot map (pic_compose), the re-rotation and stitching of the documents
// (pic_relocate) and the inline append of one layer (pic_append_inline).
//
// SemPIC, "Background: Position-Independent Caching" (Eqs. 1-3) and appendix
// "Position-Independent Linking": at link time every logical position of P,
// D_1..D_m, Q is tied to its cache slot, document keys are moved from their
// base to their final positions by R(delta), values are copied, and the
// inline tokens are rotated at their own positions.
//
// Grid x: CTA x takes the slice x of kTok positions (one page, or two when a
// token's K row is under 1024 elements, as in pic_relocate) and, with an
// append, inline token slot x; y: request.  Each CTA derives the part of the
// layout it needs by itself -- the request's document offsets (a block scan
// over at most kMaxLinkDocs lengths) and the block-table entries it needs --
// so nothing waits for another kernel: the three separate calls cost three
// chains of dependent memory round trips and two kernel boundaries, this one a
// single chain.  A CTA issues its inline token's q/k/v loads first, writes
// the layout outputs of its page (slot map, token map; the first CTA also
// the per-document offsets and deltas, the inline positions and ctx_len)
// exactly as pic_compose does, rotates and stores its token as
// pic_append_inline does, then relocates the document positions of its page
// for every layer in turn as pic_relocate does (the layout is derived once
// per page, not per layer).  Same arithmetic, same helpers: results are
// bit-identical to the three calls.  Folding the token slots into the page
// CTAs keeps a one-layer link of a few thousand positions within one wave.
#include "pic_internal.cuh"

namespace pic {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxLinkDocs = 256;   // documents per request handled in one launch
constexpr int kBM = 128;            // rows per query tile of the packed-Q workspace
constexpr int UV = 8, UK = 4;       // relocate tasks per thread per round (V, K)

struct LinkArgs {
  int batch, max_docs, n_pool, max_pages, max_ctx, max_inline, layer_begin, layer_end;
  int append_layer;  // -1: no append
  int hq, hkv, G, R_pad, t_slots, n_pages;
  long long num_pages, pool_tokens;
  const int32_t *doc_len, *doc_base, *ids, *num_docs, *spans, *prefix, *query, *block_table,
      *inline_len;
  const int64_t *doc_start;
  int32_t *doc_offset, *doc_delta, *inline_pos, *ctx_len;
  int64_t *slot_mapping, *tok_map;
  const __nv_bfloat16 *k_pool, *v_pool, *q, *k_new, *v_new;  // q/k/v_new at the append layer
  __nv_bfloat16 *k_cache, *v_cache, *qpack;
  int32_t *status;
};

__device__ long long scan256(long long v, long long *warp_tot) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const long long t = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += t;
  }
  if (lane == 31) warp_tot[warp] = v;
  __syncthreads();
  long long add = 0;
  for (int w = 0; w < warp; ++w) add += warp_tot[w];
  __syncthreads();
  return v + add;
}

// Rotate and store one 8-pair chunk held in registers (same arithmetic as
// rotate_chunk, which loads its own operands).
PIC_DEV void rot_store8(uint4 xa, uint4 xb, int c, int half, int style, const float2 *cs,
                        __nv_bfloat16 *dst) {
  float x[8], y[8], u[8], w[8];
  unpack8(xa, x);
  unpack8(xb, y);
  if (style == PIC_ROPE_HALF) {
#pragma unroll
    for (int i = 0; i < 8; ++i) { u[i] = x[i]; w[i] = y[i]; }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      u[i] = x[2 * i]; w[i] = x[2 * i + 1];
      u[4 + i] = y[2 * i]; w[4 + i] = y[2 * i + 1];
    }
  }
  rotate8(u, w, cs);
  if (style == PIC_ROPE_HALF) {
#pragma unroll
    for (int i = 0; i < 8; ++i) { x[i] = u[i]; y[i] = w[i]; }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      x[2 * i] = u[i]; x[2 * i + 1] = w[i];
      y[2 * i] = u[4 + i]; y[2 * i + 1] = w[4 + i];
    }
  }
  const PairChunk pc = pair_chunk(c, half, style);
  st_global16(dst + pc.off_a, pack8(x));
  st_global16(dst + pc.off_b, pack8(y));
}

// Shared memory of one CTA's view of its request.
struct ReqView {
  long long warp_tot[kThreads / 32];
  int off[kMaxLinkDocs];
  long long start[kMaxLinkDocs];
  int delta[kMaxLinkDocs];
  int len[kMaxLinkDocs];   // document length
  int sin[kMaxLinkDocs];   // inline index of the first token of the span after the document
  long long total;         // document and span tokens
  long long n_span;        // span tokens
  int err;
};

// Document offsets and deltas of request b (block scans over the document and
// span lengths, m <= kThreads), with pic_compose's checks; the lead CTA
// writes doc_offset / doc_delta.  Returns ctx (P + document and span tokens +
// Tq); rv.err holds the first check failed.
__device__ long long request_view(const LinkArgs &a, int b, int P, int Tq, int m, bool lead,
                                  ReqView &rv) {
  const int tid = threadIdx.x;
  long long n = 0, sp = 0, base = 0, start = 0;
  if (tid < m) {
    const int id = a.ids[(size_t)b * a.max_docs + tid];
    if (a.spans) {
      sp = a.spans[(size_t)b * a.max_docs + tid];
      if (sp < 0) {
        atomicCAS(&rv.err, 0, PIC_DEV_BAD_REQUEST);
        sp = 0;
      }
    }
    if (id < 0 || id >= a.n_pool) {
      atomicCAS(&rv.err, 0, PIC_DEV_BAD_DOC_ID);
    } else {
      n = a.doc_len[id];
      base = a.doc_base[id];
      start = a.doc_start[id];
      if (n <= 0) {
        atomicCAS(&rv.err, 0, PIC_DEV_BAD_DOC_LEN);
        n = 0;
      }
    }
  }
  const long long incl = scan256(n + sp, rv.warp_tot);
  const long long off = P + incl - (n + sp);
  const long long sincl = scan256(sp, rv.warp_tot);
  if (tid < m) {
    rv.off[tid] = (int32_t)off;
    rv.start[tid] = start;
    rv.delta[tid] = (int32_t)(off - base);
    rv.len[tid] = (int32_t)n;
    rv.sin[tid] = (int32_t)(P + sincl - sp);
    if (lead) {
      a.doc_offset[(size_t)b * a.max_docs + tid] = (int32_t)off;
      a.doc_delta[(size_t)b * a.max_docs + tid] = (int32_t)(off - base);
    }
  }
  if (tid == kThreads - 1) {
    rv.total = incl;
    rv.n_span = sincl;
  }
  if (lead)
    for (int k = m + tid; k < a.max_docs; k += kThreads) {
      a.doc_offset[(size_t)b * a.max_docs + k] = -1;
      a.doc_delta[(size_t)b * a.max_docs + k] = 0;
    }
  __syncthreads();
  const long long ctx = (long long)P + rv.total + Tq;
  if (tid == 0) {
    if (ctx > a.max_ctx || P + rv.n_span + Tq > a.max_inline)
      atomicCAS(&rv.err, 0, PIC_DEV_CTX_OVERFLOW);
    else if ((ctx + 15) / 16 > a.max_pages) atomicCAS(&rv.err, 0, PIC_DEV_BLOCK_TABLE_SHORT);
  }
  __syncthreads();
  return ctx;
}

// Logical position of inline token i of the request (prefix, spans S_1..S_m,
// query in this order), -1 past the inline tokens.
__device__ int inline_position(const ReqView &rv, int i, int P, int Tq, int m, long long ctx) {
  if (i < P) return i;
  if (i < P + rv.n_span) {  // the last span starting at or before i holds it
    int lo = 0, hi = m - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (rv.sin[mid] <= i) lo = mid;
      else hi = mid - 1;
    }
    return rv.off[lo] + rv.len[lo] + (i - rv.sin[lo]);
  }
  if (i < P + rv.n_span + Tq) return (int)(ctx - Tq + (i - P - rv.n_span));
  return -1;
}

// One inline token slot of the append layer (pic_append_inline's work), in
// two halves: its loads go out at the start of the CTA, before the token's
// position is known; its rotation and stores follow once the layout is.
struct TokLoads {
  uint4 qa, qb, ka, kb, vv;
};

template <int D>
__device__ void token_load(const LinkArgs &a, const RopeParams &rp, int b, int t, TokLoads &r) {
  constexpr int HALF = D / 2, KC = D / 16, VC = D / 8;
  const int tid = threadIdx.x;
  const size_t hkv = a.hkv, tok = (size_t)b * a.max_inline + t;
  const int nQ = a.hq * KC, nK = (int)hkv * KC, nV = (int)hkv * VC;
  r.qa = r.qb = r.ka = r.kb = r.vv = make_uint4(0, 0, 0, 0);
  const PairChunk pq = pair_chunk(tid % KC, HALF, rp.style);
  if (tid < nQ) {
    const __nv_bfloat16 *src = a.q + (tok * a.hq + tid / KC) * D;
    r.qa = ld_stream(src + pq.off_a);
    r.qb = ld_stream(src + pq.off_b);
  }
  if (tid < nK) {
    const __nv_bfloat16 *src = a.k_new + (tok * hkv + tid / KC) * D;
    r.ka = ld_stream(src + pq.off_a);
    r.kb = ld_stream(src + pq.off_b);
  }
  if (tid < nV) r.vv = ld_stream(a.v_new + (tok * hkv + tid / VC) * D + (tid % VC) * 8);
}

// Token t at logical position pos (-1: none) and cache slot `slot` (-1: none),
// cos/sin of pos in cs: R(pos) q into the packed-query workspace, R(pos) k and
// v into the cache of `layer`.
template <int D>
__device__ void token_store(const LinkArgs &a, const RopeParams &rp, int b, int layer, int t,
                            long long slot, const float2 *cs, const TokLoads &r) {
  constexpr int HALF = D / 2, KC = D / 16, VC = D / 8;
  const int tid = threadIdx.x;
  const size_t hkv = a.hkv, tok = (size_t)b * a.max_inline + t;
  const int nQ = a.hq * KC, nK = (int)hkv * KC, nV = (int)hkv * VC;
  const long long page = slot >> 4, rr = slot & 15;
  __nv_bfloat16 *kc = a.k_cache + (size_t)layer * a.num_pages * hkv * 16 * D;
  __nv_bfloat16 *vc = a.v_cache + (size_t)layer * a.num_pages * hkv * 16 * D;
  auto q_dst = [&](int h) {
    const int hk = h / a.G, g = h % a.G;
    return a.qpack + (((size_t)b * hkv + hk) * a.R_pad + (size_t)t * a.G + g) * D;
  };
  if (tid < nQ) rot_store8(r.qa, r.qb, tid % KC, HALF, rp.style, cs + 8 * (tid % KC), q_dst(tid / KC));
  if (slot >= 0) {
    if (tid < nK)
      rot_store8(r.ka, r.kb, tid % KC, HALF, rp.style, cs + 8 * (tid % KC),
                 kc + ((page * (long long)hkv + tid / KC) * 16 + rr) * D);
    if (tid < nV)
      st_global16(vc + ((page * (long long)hkv + tid / VC) * 16 + rr) * D + (tid % VC) * 8, r.vv);
  }
  for (int e = tid + kThreads; e < nQ; e += kThreads) {  // very wide models: more rounds
    const int h = e / KC, c = e % KC;
    rotate_chunk(a.q + (tok * a.hq + h) * D, q_dst(h), c, HALF, rp.style, cs + 8 * c, true);
  }
  if (slot >= 0) {
    for (int e = tid + kThreads; e < nK; e += kThreads) {
      const int h = e / KC, c = e % KC;
      rotate_chunk(a.k_new + (tok * hkv + h) * D, kc + ((page * (long long)hkv + h) * 16 + rr) * D,
                   c, HALF, rp.style, cs + 8 * c, true);
    }
    for (int e = tid + kThreads; e < nV; e += kThreads) {
      const int h = e / VC, c = e % VC;
      st_global16(vc + ((page * (long long)hkv + h) * 16 + rr) * D + c * 8,
                  ld_stream(a.v_new + (tok * hkv + h) * D + c * 8));
    }
  }
}

// Token slot t >= inline_len: zero its packed query rows.
template <int D>
__device__ void token_zero(const LinkArgs &a, int b, int t) {
  constexpr int VC = D / 8;
  for (int e = threadIdx.x; e < a.hkv * a.G * VC; e += kThreads) {
    const int hk = e / (a.G * VC), r = e % (a.G * VC), g = r / VC, c = r % VC;
    const int row = t * a.G + g;
    if (row < a.R_pad)
      st_global16(a.qpack + (((size_t)b * a.hkv + hk) * a.R_pad + row) * D + c * 8,
                  make_uint4(0, 0, 0, 0));
  }
}

// CTA x of request y: page CTA x (its kTok positions, if x < n_pages) and,
// with an append, inline token slot x (if x < t_slots).
template <int D, int kTok, bool kLayerRope>
__global__ void __launch_bounds__(kThreads) link_kernel(LinkArgs a, RopeParams rp) {
  static_assert(kTok == 16 || kTok == 32, "one warp scans the positions of a CTA");
  constexpr unsigned kMask = kTok == 32 ? 0xffffffffu : 0x0000ffffu;
  // wait for the previous kernel; the dependent launch is released later
  asm volatile("griddepcontrol.wait;" ::: "memory");
  constexpr int HALF = D / 2, KC = D / 16, VC = D / 8;
  const int b = blockIdx.y, tid = threadIdx.x;
  __shared__ ReqView rv;
  const bool has_page = (int)blockIdx.x < a.n_pages;
  const int ti = a.append_layer >= 0 && (int)blockIdx.x < a.t_slots ? (int)blockIdx.x : -1;
  const bool lead = blockIdx.x == 0;                     // per-request outputs
  const long long t0 = (long long)blockIdx.x * kTok;
  const int style = rp.style;

  __shared__ long long s_src[kTok], s_dst[kTok];
  __shared__ int s_doc[kTok];               // document index of each position
  __shared__ int s_first, s_last;
  // per touched document; with a table per layer, two buffers (this layer's
  // and the next one's, computed while this layer's loads are in flight)
  __shared__ float2 s_cs[kLayerRope ? 2 : 1][kTok][HALF];
  __shared__ float2 s_tcs[HALF];            // at the inline token's position
  __shared__ long long s_tslot;
  __shared__ int s_tpos;

  // ---- the inline token's loads (rows past inline_len are read and dropped),
  // the request scalars and the block-table entry of each position: all
  // independent of one another
  TokLoads tl;
  if (ti >= 0 && ti < a.max_inline) token_load<D>(a, rp, b, ti, tl);
  const int P = a.prefix[b], Tq = a.query[b], m = a.num_docs[b];
  const long long pidx = (t0 + tid) / 16;
  const int page_raw = has_page && tid < kTok && pidx < a.max_pages
                           ? a.block_table[(size_t)b * a.max_pages + pidx] : -1;
  const int tin = a.inline_len ? min(max(a.inline_len[b], 0), a.max_inline) : 0;
  if (tid == 0) {
    rv.err = 0;
    s_first = -1;
  }
  __syncthreads();
  if (P < 0 || Tq < 0 || m < 0 || m > a.max_docs || m > kMaxLinkDocs) {
    if (lead && tid == 0) {
      dev_fail(a.status, PIC_DEV_BAD_REQUEST, b);
      a.ctx_len[b] = -1;
    }
    return;
  }
  const long long ctx = request_view(a, b, P, Tq, m, lead, rv);
  const long long span_end = ctx - Tq;  // documents and spans occupy [P, span_end)
  const int err_view = rv.err;          // the document and size checks
  // more inline tokens than prefix, spans and query: reported by the lead CTA
  const bool bad_tin = lead && a.append_layer >= 0 && tin > P + rv.n_span + Tq;
  const int err = err_view ? err_view : (bad_tin ? PIC_DEV_BAD_POSITION : 0);

  // ---- the inline token's position and slot (one thread of warp 1)
  if (ti >= 0 && tid == 32) {
    int pos = -1;
    long long slot = -1;
    if (ti < tin) {
      if (!err_view) pos = inline_position(rv, ti, P, Tq, m, ctx);
      if (pos < 0 || pos >= a.max_ctx) {
        if (!err_view) dev_fail(a.status, PIC_DEV_BAD_POSITION, b);
        pos = -1;
      } else {
        const int page = a.block_table[(size_t)b * a.max_pages + pos / 16];
        if (page < 0 || page >= a.num_pages) dev_fail(a.status, PIC_DEV_BAD_PAGE, b);
        else slot = (long long)page * 16 + pos % 16;
      }
    }
    s_tpos = pos;
    s_tslot = slot;
  }

  // ---- this page: slot, token map, document of each position (warp 0)
  if (has_page && tid < kTok) {
    const long long t = t0 + tid;
    long long sl = -1, tm = -1, src = -1;
    int k = 0;
    if (t < a.max_ctx && !err && t < ctx) {
      if (page_raw < 0 || page_raw >= a.num_pages) atomicCAS(&rv.err, 0, PIC_DEV_BAD_PAGE);
      else sl = (long long)page_raw * 16 + t % 16;
      if (t >= P && t < span_end) {  // last document whose offset <= t; its token unless in its span
        int lo = 0, hi = m - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (rv.off[mid] <= t) lo = mid;
          else hi = mid - 1;
        }
        if (t < (long long)rv.off[lo] + rv.len[lo]) {
          k = lo;
          src = rv.start[lo] + (t - rv.off[lo]);
          tm = ((long long)lo << 40) | src;
        }
      }
    }
    if (t < a.max_ctx) {
      a.slot_mapping[(size_t)b * a.max_ctx + t] = sl;
      a.tok_map[(size_t)b * a.max_ctx + t] = tm;
    }
    // relocation source: a document token with a valid slot and pool row
    if (tm >= 0 && (src >= a.pool_tokens || k >= a.max_docs)) {
      atomicCAS(&rv.err, 0, PIC_DEV_BAD_DOC_LEN);
      src = -1;
    }
    if (sl < 0) src = -1;
    s_src[tid] = tm >= 0 ? src : -1;
    s_dst[tid] = sl;
    s_doc[tid] = k;
    const unsigned valid = __ballot_sync(kMask, s_src[tid] >= 0);
    const int kf = __shfl_sync(kMask, k, valid ? __ffs(valid) - 1 : 0);
    const int kl = __shfl_sync(kMask, k, valid ? 31 - __clz(valid) : 0);
    if (tid == 0) {
      s_first = valid ? kf : -1;
      s_last = valid ? kl : -1;
    }
  }
  if (lead) {
    int32_t *ip = a.inline_pos + (size_t)b * a.max_inline;
    for (int i = tid; i < a.max_inline; i += kThreads)
      ip[i] = err ? -1 : inline_position(rv, i, P, Tq, m, ctx);
  }
  __syncthreads();
  const size_t hkv = a.hkv;

  // ---- cos/sin at the token's position and of the documents this page touches
  if (ti >= 0 && ti < tin)
    for (int i = tid; i < HALF; i += kThreads)
      s_tcs[i] = rope_cos_sin(max(s_tpos, 0), rope_theta(rp, a.append_layer, i));
  const int k_first = s_first;
  const int n_docs = k_first >= 0 ? min(s_last - s_first + 1, kTok) : 0;
  auto fill_cs = [&](int layer, int buf) {  // cos/sin of the documents this page touches
    for (int e = tid; e < n_docs * HALF; e += kThreads) {
      const int j = e / HALF, i = e % HALF;
      const long long dl = rv.delta[k_first + j];
      s_cs[buf][j][i] = kLayerRope ? rope_cos_sin_fast(dl, rope_theta(rp, layer, i))
                                   : rope_cos_sin(dl, rope_theta(rp, layer, i));
    }
  };
  fill_cs(a.layer_begin, 0);
  __syncthreads();

  // ---- the inline token: R(p) q packed, R(p) k and v into the cache
  if (ti >= 0) {
    if (ti < tin) token_store<D>(a, rp, b, a.append_layer, ti, s_tslot, s_tcs, tl);
    else token_zero<D>(a, b, ti);
  }

  // The next kernel (attention) may be launched once every CTA got here: a
  // release at the start of the kernel made a one-layer pass slower (its
  // CTAs were then placed while this kernel still set up), one at the end
  // gave away the overlap with this kernel's last stores.
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  // ---- relocate the document positions of this page, layer by layer (with
  // a rotary table per layer, the cos/sin are recomputed for each layer;
  // that form is a separate instantiation so the common one keeps its
  // tighter loop)
  if (k_first >= 0) {
    for (int layer = a.layer_begin; layer < a.layer_end; ++layer) {
    const int cur = kLayerRope ? (layer - a.layer_begin) & 1 : 0;
    const __nv_bfloat16 *kp = a.k_pool + (size_t)layer * a.pool_tokens * hkv * D;
    const __nv_bfloat16 *vp = a.v_pool + (size_t)layer * a.pool_tokens * hkv * D;
    __nv_bfloat16 *kc = a.k_cache + (size_t)layer * a.num_pages * hkv * 16 * D;
    __nv_bfloat16 *vc = a.v_cache + (size_t)layer * a.num_pages * hkv * 16 * D;
    const int nV = kTok * (int)hkv * VC, nK = kTok * (int)hkv * KC;
    for (int round = 0; round * kThreads * UV < nV || round * kThreads * UK < nK; ++round) {
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
#pragma unroll
      for (int u = 0; u < UV; ++u)
        if (vdst[u] >= 0) st_global16(vc + vdst[u], v[u]);
#pragma unroll
      for (int u = 0; u < UK; ++u)
        if (kdst[u] >= 0)
          rot_store8(ka[u], kb[u], kch[u], HALF, style, &s_cs[cur][kdoc[u]][8 * kch[u]],
                     kc + kdst[u]);
    }
    if constexpr (kLayerRope) __syncthreads();  // next table written; this one read
    }
  }

  __syncthreads();
  const int fin = rv.err ? rv.err : (bad_tin ? PIC_DEV_BAD_POSITION : 0);
  if (tid == 0 && fin) dev_fail(a.status, fin, b);
  if (lead && tid == 0) a.ctx_len[b] = fin ? -1 : (int32_t)ctx;
}

}  // namespace
}  // namespace pic

extern "C" pic_status_t pic_link(
    const pic_geom_t *geom, int32_t batch, int32_t max_docs, int32_t n_pool_docs,
    const int32_t *doc_len, const int32_t *doc_base_pos, const int64_t *doc_token_start,
    const int32_t *req_doc_ids, const int32_t *req_num_docs, const int32_t *span_len,
    const int32_t *prefix_len, const int32_t *query_len, const int32_t *block_table,
    int32_t max_pages, int64_t num_pages,
    int32_t max_ctx, int32_t max_inline, const void *k_pool, const void *v_pool,
    int64_t pool_tokens, int32_t layer_begin, int32_t layer_end, int32_t append_layer,
    const void *q, const void *k_new, const void *v_new, const int32_t *inline_len,
    void *k_cache, void *v_cache, int32_t *doc_offset, int32_t *doc_delta,
    int64_t *slot_mapping, int64_t *tok_map, int32_t *inline_pos, int32_t *ctx_len,
    void *workspace, size_t workspace_bytes, pic_stream_t stream) {
  using namespace pic;
  RopeParams rp;
  pic_status_t st = make_rope(geom, &rp);
  if (st != PIC_OK) return st;
  if (batch <= 0 || max_docs < 0 || n_pool_docs < 0 || max_pages <= 0 || num_pages <= 0 ||
      max_ctx <= 0 || max_inline <= 0)
    return fail(PIC_ERR_INVALID_ARG, "pic_link: sizes must be positive");
  if (layer_begin < 0 || layer_end > geom->num_layers || layer_begin >= layer_end)
    return fail(PIC_ERR_INVALID_ARG, "pic_link: layer range [%d, %d) outside [0, %d)", layer_begin,
                layer_end, geom->num_layers);
  const bool do_append = append_layer >= 0;
  if (do_append && (append_layer < layer_begin || append_layer >= layer_end))
    return fail(PIC_ERR_INVALID_ARG, "pic_link: append layer %d outside [%d, %d)", append_layer,
                layer_begin, layer_end);
  if (!doc_len || !doc_base_pos || !doc_token_start || !req_num_docs || !prefix_len ||
      !query_len || !block_table || !slot_mapping || !tok_map || !inline_pos || !ctx_len ||
      (max_docs > 0 && (!req_doc_ids || !doc_offset || !doc_delta || !k_pool || !v_pool)) ||
      !k_cache || !v_cache || (do_append && (!q || !k_new || !v_new || !inline_len || !workspace)))
    return fail(PIC_ERR_INVALID_ARG, "pic_link: NULL tensor");

  // More documents per request than one CTA scans: the three calls in order.
  if (max_docs > kMaxLinkDocs || max_docs == 0) {
    st = pic_compose(geom, batch, max_docs, n_pool_docs, doc_len, doc_base_pos, doc_token_start,
                     req_doc_ids, req_num_docs, span_len, prefix_len, query_len, block_table,
                     max_pages,
                     num_pages, max_ctx, max_inline, doc_offset, doc_delta, slot_mapping, tok_map,
                     inline_pos, ctx_len, stream);
    if (st == PIC_OK && max_docs > 0)
      st = pic_relocate_mapped(geom, batch, max_docs, k_pool, v_pool, pool_tokens, tok_map, doc_delta,
                        slot_mapping, max_ctx, num_pages, k_cache, v_cache, layer_begin, layer_end,
                        stream);
    if (st == PIC_OK && do_append)
      st = pic_append_inline(geom, append_layer, batch, max_inline, q, k_new, v_new, inline_pos,
                             inline_len, slot_mapping, max_ctx, num_pages, k_cache, v_cache,
                             workspace, workspace_bytes, stream);
    return st;
  }

  if (num_pages > (int64_t)INT32_MAX)
    return fail(PIC_ERR_INVALID_ARG, "pic_link: num_pages exceeds int32");
  if (pool_tokens <= 0 || pool_tokens >= (1LL << 40))
    return fail(PIC_ERR_UNSUPPORTED, "pic_link: pool rows outside (0, 2^40)");
  if (layer_end - layer_begin > 65535 || batch > 65535)
    return fail(PIC_ERR_INVALID_ARG, "pic_link: grid too large");
  if ((reinterpret_cast<uintptr_t>(k_pool) | reinterpret_cast<uintptr_t>(v_pool) |
       reinterpret_cast<uintptr_t>(k_cache) | reinterpret_cast<uintptr_t>(v_cache) |
       reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k_new) |
       reinterpret_cast<uintptr_t>(v_new) | reinterpret_cast<uintptr_t>(workspace)) & 15)
    return fail(PIC_ERR_INVALID_ARG, "pic_link: bf16 tensors must be 16-byte aligned");
  const int G = geom->num_q_heads / geom->num_kv_heads;
  // packed-query layout of the prefill workspace (as pic_append_inline writes it)
  const int m_tiles = (int)(((long long)max_inline * G + kBM - 1) / kBM);
  const int R_pad = m_tiles * kBM;
  const size_t q_bytes = (size_t)batch * geom->num_kv_heads * R_pad * geom->head_dim * 2;
  if (do_append && workspace_bytes < q_bytes)
    return fail(PIC_ERR_WORKSPACE, "pic_link: workspace needs %zu bytes for the packed queries",
                q_bytes);
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_link: no device status word");

  LinkArgs a;
  a.batch = batch;
  a.max_docs = max_docs;
  a.n_pool = n_pool_docs;
  a.max_pages = max_pages;
  a.max_ctx = max_ctx;
  a.max_inline = max_inline;
  a.layer_begin = layer_begin;
  a.layer_end = layer_end;
  a.append_layer = do_append ? append_layer : -1;
  a.hq = geom->num_q_heads;
  a.hkv = geom->num_kv_heads;
  a.G = G;
  a.R_pad = R_pad;
  a.t_slots = std::max(max_inline, (R_pad + G - 1) / G);
  // one page per CTA when a token carries >= 1024 K elements, else two
  const bool wide = geom->num_kv_heads * geom->head_dim >= 1024;
  const int tok = wide ? 16 : 32;
  a.n_pages = (max_ctx + tok - 1) / tok;
  a.num_pages = num_pages;
  a.pool_tokens = pool_tokens;
  a.doc_len = doc_len;
  a.doc_base = doc_base_pos;
  a.ids = req_doc_ids;
  a.num_docs = req_num_docs;
  a.spans = max_docs > 0 ? span_len : nullptr;
  a.prefix = prefix_len;
  a.query = query_len;
  a.block_table = block_table;
  a.inline_len = do_append ? inline_len : nullptr;
  a.doc_start = doc_token_start;
  a.doc_offset = doc_offset;
  a.doc_delta = doc_delta;
  a.inline_pos = inline_pos;
  a.ctx_len = ctx_len;
  a.slot_mapping = slot_mapping;
  a.tok_map = tok_map;
  a.k_pool = static_cast<const __nv_bfloat16 *>(k_pool);
  a.v_pool = static_cast<const __nv_bfloat16 *>(v_pool);
  a.q = static_cast<const __nv_bfloat16 *>(q);
  a.k_new = static_cast<const __nv_bfloat16 *>(k_new);
  a.v_new = static_cast<const __nv_bfloat16 *>(v_new);
  a.k_cache = static_cast<__nv_bfloat16 *>(k_cache);
  a.v_cache = static_cast<__nv_bfloat16 *>(v_cache);
  a.qpack = static_cast<__nv_bfloat16 *>(workspace);
  a.status = status;

  dim3 grid((unsigned)(do_append ? std::max(a.n_pages, a.t_slots) : a.n_pages), batch);
  const dim3 block(kThreads);
  cudaError_t e;
  const bool per_layer = rp.layer_theta != nullptr;
  if (geom->head_dim == 128) {
    if (per_layer)
      e = wide ? launch_dependent(link_kernel<128, 16, true>, grid, block, 0, stream, a, rp)
               : launch_dependent(link_kernel<128, 32, true>, grid, block, 0, stream, a, rp);
    else
      e = wide ? launch_dependent(link_kernel<128, 16, false>, grid, block, 0, stream, a, rp)
               : launch_dependent(link_kernel<128, 32, false>, grid, block, 0, stream, a, rp);
  } else {
    if (per_layer)
      e = wide ? launch_dependent(link_kernel<64, 16, true>, grid, block, 0, stream, a, rp)
               : launch_dependent(link_kernel<64, 32, true>, grid, block, 0, stream, a, rp);
    else
      e = wide ? launch_dependent(link_kernel<64, 16, false>, grid, block, 0, stream, a, rp)
               : launch_dependent(link_kernel<64, 32, false>, grid, block, 0, stream, a, rp);
  }
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, "pic_link launch");
  return PIC_OK;
}
