// Bulk copy by SM loads and stores, for moving a step's inputs from pinned host memory
// to the device (and results back).  On a Grace-Blackwell node a kernel reading pinned
// host memory through unified addressing streams it over NVLink-C2C about twice as fast
// as the copy engines; the same kernel also copies device to device.
#include "netkv_internal.cuh"

namespace {

__global__ void __launch_bounds__(512) copy_kernel(const uint4* __restrict__ src,
                                                   uint4* __restrict__ dst, size_t n16,
                                                   const unsigned char* __restrict__ src_tail,
                                                   unsigned char* __restrict__ dst_tail,
                                                   size_t tail) {
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  const size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (size_t i = t; i < n16; i += stride) dst[i] = __ldcs(src + i);
  if (t < tail) dst_tail[t] = src_tail[t];
}

}  // namespace

extern "C" netkv_status netkv_copy_async(void* dst, const void* src, size_t bytes,
                                         netkv_stream_t stream) {
  if (bytes == 0) return NETKV_OK;
  if (!dst || !src || !aligned_to(dst, 16) || !aligned_to(src, 16)) return NETKV_EINVAL;
  int dev = 0, sms = 0;
  NETKV_CUDA_TRY(cudaGetDevice(&dev));
  NETKV_CUDA_TRY(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const size_t n16 = bytes / 16, tail = bytes % 16;
  const size_t want = (n16 + 511) / 512;
  const unsigned grid = (unsigned)(want < (size_t)sms * 4 ? (want ? want : 1) : (size_t)sms * 4);
  copy_kernel<<<grid, 512, 0, (cudaStream_t)stream>>>(
      reinterpret_cast<const uint4*>(src), reinterpret_cast<uint4*>(dst), n16,
      reinterpret_cast<const unsigned char*>(src) + n16 * 16,
      reinterpret_cast<unsigned char*>(dst) + n16 * 16, tail);
  return netkv_launch_status();
}
