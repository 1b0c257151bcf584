// Library-wide plumbing of libpic: error strings, the per-device status word,
// geometry checks and TMA descriptor encoding.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "pic_internal.cuh"

namespace pic {

// {code, detail} of the first device-side failure since the last read.
__device__ int32_t g_device_status[2];

static thread_local char t_last_error[512] = "";

pic_status_t fail(pic_status_t s, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(t_last_error, sizeof(t_last_error), fmt, ap);
  va_end(ap);
  return s;
}

pic_status_t cuda_fail(cudaError_t e, const char *what) {
  return fail(PIC_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

void *device_address(const void *p) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();  // clear the error the failed query recorded
    return nullptr;
  }
  switch (at.type) {
    case cudaMemoryTypeDevice:
      return at.device == dev ? const_cast<void *>(p) : nullptr;
    case cudaMemoryTypeHost:
    case cudaMemoryTypeManaged:
      return at.devicePointer;
    default:
      return nullptr;
  }
}

unsigned long long current_context_id() {
  using GetCurrentFn = CUresult (*)(CUcontext *);
  using GetIdFn = CUresult (*)(CUcontext, unsigned long long *);
  static GetCurrentFn get_current = nullptr;
  static GetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetIdFn>(p);
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx ||
      get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

int32_t *device_status_ptr() {
  constexpr int kMaxDev = 64;
  static int32_t *ptrs[kMaxDev] = {nullptr};
  static unsigned long long ctx_ids[kMaxDev] = {0};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return nullptr;
  std::lock_guard<std::mutex> lk(mu);
  // looked up once per device context: a device reset makes a new context
  // (and a new copy of the word), so the address is looked up again
  const unsigned long long id = current_context_id();
  if (!ptrs[dev] || id == 0 || id != ctx_ids[dev]) {
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_status) != cudaSuccess) return nullptr;
    ptrs[dev] = static_cast<int32_t *>(p);
    ctx_ids[dev] = current_context_id();
  }
  return ptrs[dev];
}

pic_status_t check_geom(const pic_geom_t *g, double *theta) {
  if (!g) return fail(PIC_ERR_INVALID_ARG, "geometry is NULL");
  if (g->num_layers <= 0 || g->num_q_heads <= 0 || g->num_kv_heads <= 0)
    return fail(PIC_ERR_INVALID_ARG, "layers/heads must be positive");
  if (g->num_q_heads % g->num_kv_heads)
    return fail(PIC_ERR_INVALID_ARG, "num_q_heads %d is not a multiple of num_kv_heads %d",
                g->num_q_heads, g->num_kv_heads);
  if (g->head_dim != 64 && g->head_dim != 128)
    return fail(PIC_ERR_UNSUPPORTED, "head_dim %d (supported: 64, 128)", g->head_dim);
  if (g->page_size != 16) return fail(PIC_ERR_UNSUPPORTED, "page_size %d (supported: 16)", g->page_size);
  if (g->rope_style != PIC_ROPE_HALF && g->rope_style != PIC_ROPE_INTERLEAVED)
    return fail(PIC_ERR_INVALID_ARG, "rope_style %d", g->rope_style);
  const int half = g->head_dim / 2;
  if (g->inv_freq) {
    for (int i = 0; i < half; ++i) {
      if (!(g->inv_freq[i] > 0.0) || !std::isfinite(g->inv_freq[i]))
        return fail(PIC_ERR_INVALID_ARG, "inv_freq[%d] must be positive and finite", i);
      theta[i] = g->inv_freq[i];
    }
  } else {
    if (!(g->rope_base > 1.0) || !std::isfinite(g->rope_base))
      return fail(PIC_ERR_INVALID_ARG, "rope_base must be > 1");
    for (int i = 0; i < half; ++i)
      theta[i] = std::pow(g->rope_base, -2.0 * (double)i / (double)g->head_dim);
  }
  for (int i = half; i < kMaxHalfDim; ++i) theta[i] = 0.0;
  return PIC_OK;
}

using EncodeFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                              const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                              const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeFn get_encode() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

pic_status_t encode_tmap_2d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t rows,
                            uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows) {
  EncodeFn enc = get_encode();
  if (!enc) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (row_stride_bytes & 15))
    return fail(PIC_ERR_INVALID_ARG, "tensor base/stride not 16-byte aligned");
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {row_stride_bytes};
  cuuint32_t box[2] = {box_inner, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims,
                   strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
  return PIC_OK;
}

pic_status_t encode_tmap_3d(CUtensorMap *map, const void *base, uint64_t inner, uint64_t mid,
                            uint64_t outer, uint64_t mid_stride_bytes, uint64_t outer_stride_bytes,
                            uint32_t box_inner, uint32_t box_mid, uint32_t box_outer) {
  EncodeFn enc = get_encode();
  if (!enc) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (mid_stride_bytes & 15) || (outer_stride_bytes & 15))
    return fail(PIC_ERR_INVALID_ARG, "tensor base/strides not 16-byte aligned");
  cuuint64_t dims[3] = {inner, mid, outer};
  cuuint64_t strides[2] = {mid_stride_bytes, outer_stride_bytes};
  cuuint32_t box[3] = {box_inner, box_mid, box_outer};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims,
                   strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled (3d) failed (%d)", (int)r);
  return PIC_OK;
}

pic_status_t encode_tmap_pool128(CUtensorMap *map, const void *base, uint64_t rows, int hkv) {
  EncodeFn enc = get_encode();
  if (!enc) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  if (reinterpret_cast<uintptr_t>(base) & 15)
    return fail(PIC_ERR_INVALID_ARG, "tensor base not 16-byte aligned");
  if (rows <= 16) return fail(PIC_ERR_INVALID_ARG, "pool has too few rows for a page box");
  const uint64_t row_bytes = (uint64_t)hkv * 128 * 2;
  // {column, row, panel, 8-row half, head}: a box at row R covers rows R..R+7
  // (half 0) and R+8..R+15 (half 1); the row extent stops 8 short of the end
  // so both halves stay inside the pool
  cuuint64_t dims[5] = {64, rows - 8, 2, 2, (cuuint64_t)hkv};
  cuuint64_t strides[4] = {row_bytes, 128, 8 * row_bytes, 256};
  cuuint32_t box[5] = {64, 8, 2, 2, 1};
  cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(base), dims,
                   strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled (pool) failed (%d)", (int)r);
  return PIC_OK;
}

pic_status_t encode_tmap_pages128(CUtensorMap *map, const void *base, uint64_t n_page_heads) {
  EncodeFn enc = get_encode();
  if (!enc) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled is unavailable");
  if (reinterpret_cast<uintptr_t>(base) & 15)
    return fail(PIC_ERR_INVALID_ARG, "tensor base not 16-byte aligned");
  cuuint64_t dims[4] = {64, 8, 2, 2 * n_page_heads};
  cuuint64_t strides[3] = {256, 128, 2048};
  cuuint32_t box[4] = {64, 8, 2, 2};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims,
                   strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(PIC_ERR_CUDA, "cuTensorMapEncodeTiled (page heads) failed (%d)", (int)r);
  return PIC_OK;
}

}  // namespace pic

extern "C" {

int32_t pic_abi_version(void) { return PIC_ABI_VERSION; }

const char *pic_last_error(void) { return pic::t_last_error; }

pic_status_t pic_device_status(pic_stream_t stream, int32_t *code, int32_t *detail) {
  int32_t *p = pic::device_status_ptr();
  if (!p) return pic::fail(PIC_ERR_CUDA, "device status word unavailable");
  int32_t host[2] = {0, 0};
  cudaError_t e = cudaMemcpyAsync(host, p, sizeof(host), cudaMemcpyDeviceToHost, stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return pic::cuda_fail(e, "pic_device_status");
  e = cudaMemsetAsync(p, 0, sizeof(host), stream);
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return pic::cuda_fail(e, "pic_device_status reset");
  if (code) *code = host[0];
  if (detail) *detail = host[1];
  if (host[0] != PIC_DEV_OK)
    return pic::fail(PIC_ERR_DEVICE, "device check failed: code %d detail %d", host[0], host[1]);
  return PIC_OK;
}

}  // extern "C"
