// pic_copy_async: host <-> device transfers of a request's inputs and
// outputs moved by the GPU's own loads and stores.  On a Grace-Blackwell
// node page-locked host memory is reachable from kernels over the coherent
// chip-to-chip link, which a kernel with many 16-byte requests in flight
// drives well above the rate the copy engines reach for transfers of a few
// megabytes.  Either side may be device memory of the current device or
// page-locked host memory (cudaHostAlloc / cudaHostRegister, e.g. a pinned
// torch tensor); the kernel addresses host memory through its device
// pointer.  Two checks of the path's machinery live here too:
// pic_launch_probe (empty programmatic-dependent kernels of given launch
// shapes, the launch floor of a pass) and pic_wait_probe (the bounded
// mbarrier wait running out and reporting PIC_DEV_TIMEOUT).
#include <algorithm>

#include "pic_internal.cuh"

namespace pic {
namespace {

constexpr int kCopyThreads = 256;
constexpr int kCopyUnroll = 4;  // 16-byte loads in flight per thread

// dst[i] = src[i] for i < n16 (16-byte words), then the tail bytes.
__global__ void __launch_bounds__(kCopyThreads) copy_kernel(uint4 *__restrict__ dst,
                                                            const uint4 *__restrict__ src,
                                                            size_t n16, uint8_t *__restrict__ dst_tail,
                                                            const uint8_t *__restrict__ src_tail,
                                                            int tail) {
  const size_t per_block = (size_t)kCopyThreads * kCopyUnroll;
  const size_t stride = (size_t)gridDim.x * per_block;
  for (size_t base = (size_t)blockIdx.x * per_block + threadIdx.x; base < n16; base += stride) {
    uint4 v[kCopyUnroll];
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) {
      const size_t k = base + (size_t)u * kCopyThreads;
      if (k < n16) v[u] = src[k];
    }
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) {
      const size_t k = base + (size_t)u * kCopyThreads;
      if (k < n16) dst[k] = v[u];
    }
  }
  if (blockIdx.x == 0 && (int)threadIdx.x < tail) dst_tail[threadIdx.x] = src_tail[threadIdx.x];
}

// An empty programmatic dependent: waits for the kernel before, lets the
// next one launch, and does nothing else (pic_launch_probe).
__global__ void probe_kernel() { pdl_entry(); }

// One CTA waits on the first phase of an mbarrier of one arrival with the
// bounded wait of the path's kernels (pic_wait_probe): thread 0 arrives
// first when `arrive` is set, so the wait completes at once; otherwise
// nothing arrives, the wait runs out after limit_ns and records
// PIC_DEV_TIMEOUT (detail -1) in the status word, and the kernel returns.
__global__ void wait_probe_kernel(int arrive, uint64_t limit_ns, int32_t *status) {
  __shared__ __align__(8) uint64_t bar_slot;
  __shared__ int abort_flag;
  const uint32_t bar = smem_u32(&bar_slot);
  if (threadIdx.x == 0) {
    mbar_init(bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (arrive) mbar_arrive(bar);
    mbar_wait_for(bar, 0, &abort_flag, status, -1, limit_ns);
  }
  __syncthreads();
}

}  // namespace
}  // namespace pic

extern "C" pic_status_t pic_wait_probe(int32_t arrive, int64_t limit_ns, pic_stream_t stream) {
  using namespace pic;
  if (limit_ns < 1000 || limit_ns > 10000000000LL)
    return fail(PIC_ERR_INVALID_ARG, "pic_wait_probe: limit_ns outside [1 us, 10 s]");
  int32_t *status = device_status_ptr();
  if (!status) return fail(PIC_ERR_CUDA, "pic_wait_probe: no device status word");
  wait_probe_kernel<<<1, 32, 0, stream>>>(arrive != 0, (uint64_t)limit_ns, status);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? PIC_OK : cuda_fail(e, "pic_wait_probe launch");
}

extern "C" pic_status_t pic_launch_probe(int32_t n, const int32_t *grid, const int32_t *block,
                                         const int32_t *smem, pic_stream_t stream) {
  using namespace pic;
  if (n <= 0 || !grid || !block || !smem)
    return fail(PIC_ERR_INVALID_ARG, "pic_launch_probe: n > 0 and all arrays required");
  int dev = 0, max_smem = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return cuda_fail(e, "pic_launch_probe: device query");
  int top = 0;
  for (int i = 0; i < n; ++i) {
    if (grid[3 * i] <= 0 || grid[3 * i + 1] <= 0 || grid[3 * i + 2] <= 0 || block[i] <= 0 ||
        block[i] > 1024 || smem[i] < 0 || smem[i] > max_smem)
      return fail(PIC_ERR_INVALID_ARG, "pic_launch_probe: launch %d out of range", i);
    top = std::max(top, (int)smem[i]);
  }
  e = cudaFuncSetAttribute(probe_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, top);
  if (e != cudaSuccess) return cuda_fail(e, "pic_launch_probe smem attribute");
  for (int i = 0; i < n; ++i) {
    e = launch_dependent(probe_kernel, dim3(grid[3 * i], grid[3 * i + 1], grid[3 * i + 2]),
                         dim3(block[i]), (size_t)smem[i], stream);
    if (e != cudaSuccess) return cuda_fail(e, "pic_launch_probe launch");
  }
  return PIC_OK;
}

extern "C" pic_status_t pic_copy_async(void *dst, const void *src, size_t bytes, pic_stream_t stream) {
  using namespace pic;
  if (bytes == 0) return PIC_OK;
  if (!dst || !src) return fail(PIC_ERR_INVALID_ARG, "pic_copy_async: NULL pointer");
  void *d = device_address(dst);
  const void *s = device_address(src);
  if (!d || !s)
    return fail(PIC_ERR_INVALID_ARG,
                "pic_copy_async: %s is neither memory of the current device nor page-locked host memory",
                !d ? "dst" : "src");
  cudaError_t e;
  const uintptr_t du = reinterpret_cast<uintptr_t>(d), su = reinterpret_cast<uintptr_t>(s);
  if (du < su ? su - du < bytes : du - su < bytes)
    return fail(PIC_ERR_INVALID_ARG, "pic_copy_async: overlapping ranges");
  if ((du | su) & 15) {
    // unaligned: the copy engine moves it
    e = cudaMemcpyAsync(d, s, bytes, cudaMemcpyDefault, stream);
    return e == cudaSuccess ? PIC_OK : cuda_fail(e, "pic_copy_async (unaligned)");
  }
  const size_t n16 = bytes / 16;
  const int tail = (int)(bytes % 16);
  const size_t per_block = (size_t)kCopyThreads * kCopyUnroll;
  const size_t blocks = std::max<size_t>(1, std::min<size_t>((n16 + per_block - 1) / per_block, 152 * 8));
  copy_kernel<<<(unsigned)blocks, kCopyThreads, 0, stream>>>(
      static_cast<uint4 *>(d), static_cast<const uint4 *>(s), n16,
      static_cast<uint8_t *>(d) + n16 * 16, static_cast<const uint8_t *>(s) + n16 * 16, tail);
  e = cudaGetLastError();
  return e == cudaSuccess ? PIC_OK : cuda_fail(e, "pic_copy_async launch");
}
