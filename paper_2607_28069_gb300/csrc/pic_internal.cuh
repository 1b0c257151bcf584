// Internal helpers shared by the kernels of libpic (never installed).
//
// Contents: host-side error reporting and geometry checks, the per-device
// status word, RoPE angle evaluation, bf16 packing, and thin inline-PTX
// wrappers for the sm_103a features the kernels use (mbarrier, TMA bulk
// tensor copies, tcgen05 MMA / TMEM, legacy warp MMA for decode).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <cmath>

#include <utility>

#include "../../include/pic.h"

namespace pic {

// ---------------------------------------------------------------- host side
pic_status_t fail(pic_status_t s, const char *fmt, ...);
pic_status_t cuda_fail(cudaError_t e, const char *what);
// The address kernels use for p: p itself for memory of the current device,
// the mapped address for page-locked (or managed) host memory; NULL for
// pageable host memory or another device's memory.
void *device_address(const void *p);
// Address of the current device's status word ({code, detail}).
int32_t *device_status_ptr();
// Unique identity of the calling thread's current CUDA context (0 when it has
// none or the driver cannot say): device addresses of module variables are
// valid for one context, and a device reset replaces it.
unsigned long long current_context_id();
// Validates the geometry and fills theta[0..d/2) (fp64 frequencies).
pic_status_t check_geom(const pic_geom_t *g, double *theta);

// RoPE parameters passed by value to kernels.
struct RopeParams {
  double theta[64];            // frequencies, d/2 <= 64
  const double *layer_theta;   // device [num_layers][d/2] per-layer frequencies, or null
  int half;                    // d / 2
  int style;                   // PIC_ROPE_HALF / PIC_ROPE_INTERLEAVED
};

inline pic_status_t make_rope(const pic_geom_t *g, RopeParams *rp) {
  pic_status_t s = check_geom(g, rp->theta);
  rp->layer_theta = g->layer_inv_freq;
  rp->half = g->head_dim / 2;
  rp->style = g->rope_style;
  return s;
}

// Document pool [L * pool_tokens][Hkv][128] bf16 as a 5-D view whose box of
// 16 consecutive rows of one head (from any row) lands like a page-head box of
// the cache: [8-row half][64-column panel][8 rows][128 B], 128-byte swizzled.
// Rows past rows - 8 read as zeros (a box always stays inside one document).
pic_status_t encode_tmap_pool128(CUtensorMap *map, const void *base, uint64_t rows, int hkv);
// cuTensorMapEncodeTiled through the runtime's driver entry point.
pic_status_t encode_tmap_2d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t rows,
                            uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows);

// Rows of `inner` elements with two strides: dims {inner, mid, outer}.
pic_status_t encode_tmap_3d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t mid,
                            uint64_t outer, uint64_t mid_stride_bytes, uint64_t outer_stride_bytes,
                            uint32_t box_inner, uint32_t box_mid, uint32_t box_outer);

// Page-head map for 128-dim caches ([..][16 rows][128 bf16] per page-head):
// 4-D view {64 columns, 8 rows, 2 column panels, 2 * n_page_heads row halves}
// with strides {256 B, 128 B, 2048 B}.  A box {64, 8, 2, 2} moves one whole
// 4 KB page-head and lands as [half][panel][8 rows][128 B], so that across a
// run of pages the 8-row groups of one panel sit at a constant 2048-byte
// stride (the SW128 operand stride) and the two panels 1024 bytes apart.
pic_status_t encode_tmap_pages128(CUtensorMap *map, const void *base, uint64_t n_page_heads);

constexpr int kMaxHalfDim = 64;

// ---------------------------------------------------------- device helpers
#define PIC_DEV __device__ __forceinline__

// Record the first device-side failure (code, detail); later ones are dropped.
PIC_DEV void dev_fail(int32_t *status, int code, int detail) {
  if (atomicCAS(status, 0, code) == 0) atomicExch(status + 1, detail);
}

// cos/sin of pos * theta: the product and its reduction to [-pi, pi] are done
// in fp64 (exact enough for |pos| up to 2^31), the final sin/cos in fp32 on
// the reduced angle, which is then accurate to a few fp32 ulps.
PIC_DEV float2 rope_cos_sin(long long pos, double theta) {
  const double two_pi = 6.283185307179586476925286766559;
  double a = (double)pos * theta;
  double k = rint(a * (1.0 / two_pi));
  double r = fma(-k, two_pi, a);
  float s, c;
  sincosf((float)r, &s, &c);
  return make_float2(c, s);
}

// The same with CUDA's fast-path sine and cosine on the reduced angle
// (|r| <= pi: absolute error about 4e-7), for tables recomputed for every
// layer of a relocation (per-layer frequencies), where the precise call
// costs more than its accuracy is worth against bf16 keys.
PIC_DEV float2 rope_cos_sin_fast(long long pos, double theta) {
  const double two_pi = 6.283185307179586476925286766559;
  double a = (double)pos * theta;
  double k = rint(a * (1.0 / two_pi));
  double r = fma(-k, two_pi, a);
  float s, c;
  __sincosf((float)r, &s, &c);
  return make_float2(c, s);
}

// Frequency i of layer `layer`: the per-layer table when the geometry has
// one, else the table shared by all layers.
PIC_DEV double rope_theta(const RopeParams &rp, int layer, int i) {
  return rp.layer_theta ? rp.layer_theta[(size_t)layer * rp.half + i] : rp.theta[i];
}

PIC_DEV void unpack8(const uint4 &v, float *f) {
  const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

PIC_DEV uint4 pack8(const float *f) {
  uint4 v;
  __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
  return v;
}

// Eight floats as fp16, rounded to nearest even and saturated at +-65504.
PIC_DEV uint4 pack8_h(const float *f) {
  uint4 v;
  __half2 *h = reinterpret_cast<__half2 *>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    h[i] = __floats2half2_rn(fminf(fmaxf(f[2 * i], -65504.f), 65504.f),
                             fminf(fmaxf(f[2 * i + 1], -65504.f), 65504.f));
  return v;
}

PIC_DEV uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&h);
}

// ---- packed fp32 pairs (one 64-bit register pair, low half first)
PIC_DEV uint64_t f2pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
PIC_DEV void f2unpack(uint64_t v, float &lo, float &hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
PIC_DEV uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t r;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
  return r;
}
PIC_DEV uint64_t mul2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
// A bf16 pair (one 32-bit word, low element first) as a packed fp32 pair (exact).
PIC_DEV uint64_t bf2_to_f2(uint32_t w) {
  uint64_t r;
  asm("{\n\t.reg .b32 lo, hi;\n\tshl.b32 lo, %1, 16;\n\tand.b32 hi, %1, 0xffff0000;\n\t"
      "mov.b64 %0, {lo, hi};\n\t}" : "=l"(r) : "r"(w));
  return r;
}
// A packed fp32 pair as a bf16 pair, each rounded to nearest even.
PIC_DEV uint32_t f2_to_bf2(uint64_t v) {
  uint32_t r;
  asm("{\n\t.reg .f32 lo, hi;\n\tmov.b64 {lo, hi}, %1;\n\tcvt.rn.bf16x2.f32 %0, hi, lo;\n\t}"
      : "=r"(r) : "l"(v));
  return r;
}
// The two halves of a packed pair, each duplicated: (lo, lo) and (hi, hi).
PIC_DEV void f2_split_dup(uint64_t v, uint64_t &lo2, uint64_t &hi2) {
  asm("{\n\t.reg .b32 lo, hi;\n\tmov.b64 {lo, hi}, %2;\n\tmov.b64 %0, {lo, lo};\n\t"
      "mov.b64 %1, {hi, hi};\n\t}" : "=l"(lo2), "=l"(hi2) : "l"(v));
}
PIC_DEV uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t r;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
  return r;
}
PIC_DEV float max3f(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// Streaming 16-byte load that bypasses L1 (each pool byte is read once).
PIC_DEV uint4 ld_stream(const void *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

PIC_DEV void st_global16(void *p, const uint4 &v) {
  asm volatile("st.global.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

// Rotate 8 RoPE pairs (u_i, w_i) by the angles whose (cos, sin) are cs[i].
PIC_DEV void rotate8(float *u, float *w, const float2 *cs) {
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    float c = cs[i].x, s = cs[i].y;
    float uu = u[i], ww = w[i];
    u[i] = fmaf(uu, c, -ww * s);
    w[i] = fmaf(uu, s, ww * c);
  }
}

// For a vector chunk c of 8 pairs, the element offsets of its two halves.
// half-split: pairs (i, i + d/2), chunk c covers i in [8c, 8c+8):
//   lo at 8c, hi at d/2 + 8c (two 16-byte pieces).
// interleaved: pairs (2i, 2i+1), chunk c covers elements [16c, 16c+16).
struct PairChunk {
  int off_a, off_b;  // element offsets of the two 16-byte pieces
};
PIC_DEV PairChunk pair_chunk(int c, int half, int style) {
  PairChunk p;
  if (style == PIC_ROPE_HALF) {
    p.off_a = 8 * c;
    p.off_b = half + 8 * c;
  } else {
    p.off_a = 16 * c;
    p.off_b = 16 * c + 8;
  }
  return p;
}

// Load / rotate / store one chunk of 8 pairs of a d-vector.
// `src`, `dst` point at the start of the d-vector; cs holds (cos, sin) of the
// 8 pairs 8c..8c+7.
// Rotates the chunk of 8 pairs whose two 16-byte halves va, vb were loaded
// from offsets pc.off_a, pc.off_b of a row, and stores it at the same
// offsets of dst.
PIC_DEV void rotate_store(uint4 va, uint4 vb, __nv_bfloat16 *dst, const PairChunk &pc, int style,
                          const float2 *cs) {
  float a[8], b[8], u[8], w[8];
  unpack8(va, a);
  unpack8(vb, b);
  if (style == PIC_ROPE_HALF) {
#pragma unroll
    for (int i = 0; i < 8; ++i) { u[i] = a[i]; w[i] = b[i]; }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      u[i] = a[2 * i]; w[i] = a[2 * i + 1];
      u[4 + i] = b[2 * i]; w[4 + i] = b[2 * i + 1];
    }
  }
  rotate8(u, w, cs);
  if (style == PIC_ROPE_HALF) {
#pragma unroll
    for (int i = 0; i < 8; ++i) { a[i] = u[i]; b[i] = w[i]; }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      a[2 * i] = u[i]; a[2 * i + 1] = w[i];
      b[2 * i] = u[4 + i]; b[2 * i + 1] = w[4 + i];
    }
  }
  st_global16(dst + pc.off_a, pack8(a));
  st_global16(dst + pc.off_b, pack8(b));
}

PIC_DEV void rotate_chunk(const __nv_bfloat16 *src, __nv_bfloat16 *dst, int c, int half,
                          int style, const float2 *cs, bool streaming) {
  const PairChunk pc = pair_chunk(c, half, style);
  const uint4 va = streaming ? ld_stream(src + pc.off_a) : *reinterpret_cast<const uint4 *>(src + pc.off_a);
  const uint4 vb = streaming ? ld_stream(src + pc.off_b) : *reinterpret_cast<const uint4 *>(src + pc.off_b);
  rotate_store(va, vb, dst, pc, style, cs);
}

PIC_DEV uint32_t smem_u32(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------------------ mbarrier
PIC_DEV void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
PIC_DEV void fence_mbar_init() { asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory"); }
PIC_DEV void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
// Programmatic dependent launch.  A kernel launched with launch_dependent()
// calls pdl_entry() first: it waits until the kernel before it on the stream
// has completed and its writes are visible (before this kernel reads or
// writes anything), then lets the next kernel's launch begin.  Because every
// kernel of a chain waits first, completion of one implies completion of all
// before it.  The next grid launches only once every CTA of this one has
// run the trigger, i.e. is resident, so it never starves this one of SMs.
PIC_DEV void pdl_entry() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                    cudaStream_t stream, Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}
// The same, with the grid in clusters of `cluster_x` consecutive CTAs along x.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block,
                                            size_t smem, cudaStream_t stream, int cluster_x,
                                            Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = (unsigned)cluster_x;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// ---- thread-block clusters
PIC_DEV uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// The shared::cluster address of `addr` (a shared::cta address of this CTA)
// in CTA `rank` of the cluster.
PIC_DEV uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
// All threads of every CTA of the cluster (release / acquire at cluster scope).
PIC_DEV void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" :::
                   "memory");
}
// One arrival on a barrier of another CTA of the cluster (`remote_bar` from
// map_to_rank), ordered after this thread's earlier memory operations.
PIC_DEV void mbar_arrive_remote(uint32_t remote_bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote_bar)
               : "memory");
}
// Bulk copy of `bytes` (a multiple of 16) from this CTA's shared memory to
// another CTA's (`dst`, `remote_bar` from map_to_rank); completes as
// transaction bytes on that CTA's barrier.
PIC_DEV void bulk_copy_to_peer(uint32_t dst, uint32_t src, uint32_t bytes, uint32_t remote_bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "r"(src), "r"(bytes), "r"(remote_bar)
      : "memory");
}

// Named CTA barriers (bar.sync / bar.arrive) shared by a fixed set of warps.
PIC_DEV void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
PIC_DEV void named_bar_arrive(int id, int nthreads) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
PIC_DEV void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
// Adds `bytes` to the barrier's expected transaction count without arriving
// (the arrival comes later, e.g. after this thread's own shared-memory writes).
PIC_DEV void mbar_expect_tx_only(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
PIC_DEV bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
PIC_DEV uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait limit for every mbarrier wait: a correct kernel waits microseconds.
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s

// Bounded wait.  Returns false (after recording PIC_DEV_TIMEOUT and raising
// *abort) when the phase did not complete within limit_ns, or when another
// role of the CTA has already aborted.
PIC_DEV bool mbar_wait_for(uint32_t bar, uint32_t parity, volatile int *abort, int32_t *status,
                           int detail, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > limit_ns) {
        *abort = 1;
        dev_fail(status, PIC_DEV_TIMEOUT, detail);
        return false;
      }
    }
  }
}
// The wait every kernel of the path uses.
PIC_DEV bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort, int32_t *status,
                       int detail) {
  return mbar_wait_for(bar, parity, abort, status, detail, kWaitLimitNs);
}

// ----------------------------------------------------------------------- TMA
PIC_DEV void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
PIC_DEV void tma_load_3d(uint32_t dst, const CUtensorMap *map, int x, int y, int z, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}
PIC_DEV void tma_load_4d(uint32_t dst, const CUtensorMap *map, int x, int y, int z, int w,
                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(bar)
      : "memory");
}
PIC_DEV void tma_load_5d(uint32_t dst, const CUtensorMap *map, int x, int y, int z, int w, int v,
                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.5d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(w), "r"(v), "r"(bar)
      : "memory");
}
PIC_DEV void prefetch_tmap(const CUtensorMap *map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
PIC_DEV void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// ------------------------------------------------------------------ tcgen05
PIC_DEV void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
}
PIC_DEV void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
PIC_DEV void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
PIC_DEV void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
PIC_DEV void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// D(tmem) (+)= A(smem desc) * B(smem desc)
PIC_DEV void mma_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                    uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D(tmem) (+)= A(tmem) * B(smem desc)
PIC_DEV void mma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                    uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on `bar` once every tcgen05 op issued so far by this thread is done.
PIC_DEV void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   bar)
               : "memory");
}
// The same commit, arriving on the barrier at this offset in every CTA of
// the cluster that `cta_mask` selects.
PIC_DEV void mma_commit_mc(uint32_t bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(bar), "h"(cta_mask)
      : "memory");
}

// 32 consecutive 32-bit TMEM columns of this thread's lane.
PIC_DEV void tmem_ld32(uint32_t taddr, uint32_t *r) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
PIC_DEV void tmem_st32(uint32_t taddr, const uint32_t *r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
PIC_DEV void tmem_st16(uint32_t taddr, const uint32_t *r) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15])
      : "memory");
}
PIC_DEV void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
PIC_DEV void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor for tcgen05.mma, 128-byte swizzle.
// start/lbo/sbo in bytes (encoded >> 4); version field 1; layout SWIZZLE_128B.
PIC_DEV uint64_t sdesc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
  d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
  d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
  d |= (uint64_t)1 << 46;
  d |= (uint64_t)2 << 61;
  return d;
}

// Instruction descriptor, kind::f16 with bf16 A/B and fp32 D.
// a_mn / b_mn: operand stored MN-major (transposed) instead of K-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) |
         ((b_mn ? 1u : 0u) << 16) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

PIC_DEV float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
PIC_DEV uint64_t exp2_mufu2(uint64_t x) {
  float x0, x1;
  f2unpack(x, x0, x1);
  return f2pack(ex2(x0), ex2(x1));
}

// --------------------------------------------------- warp MMA (decode path)
PIC_DEV void ldsm_x4(uint32_t addr, uint32_t *r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
PIC_DEV void ldsm_x4_t(uint32_t addr, uint32_t *r) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
PIC_DEV uint32_t movm_t(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
PIC_DEV void mma16816(float *d, const uint32_t *a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 16-byte shared-memory load and store (generic proxy).
PIC_DEV uint4 lds128(uint32_t addr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "r"(addr)
               : "memory");
  return v;
}
PIC_DEV void sts128(uint32_t addr, const uint4 &v) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}

// Byte offset of element (row, col) inside a [rows][64] bf16 panel written by
// TMA with 128-byte swizzle: 16-byte chunk index XOR (row mod 8).
PIC_DEV uint32_t sw128_offset(int row, int col) {
  return (uint32_t)(row * 128 + ((((col >> 3) ^ (row & 7)) << 4)) + ((col & 7) << 1));
}

}  // namespace pic
