// Transfers between device memory and page-locked host memory done by SMs
// (zarya_copy): a small grid moves 16-byte vectors through the host buffer's
// device mapping. On a Grace-Blackwell node the host link is the bound (about
// 170 GB/s for either direction measured with 16 to 304 CTAs), so a few CTAs
// suffice and the copy leaves the SMs of a concurrent step alone. As a kernel
// it joins the kernels of a CUDA graph without the copy-engine hand-over a
// memcpy node costs between kernel nodes.
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "token_ops.cuh"

namespace zarya {
namespace {

constexpr int kCopyThreads = 256;
constexpr int kCopyMaxCtas = 24;
constexpr int kCopyUnroll = 4;

__global__ void __launch_bounds__(kCopyThreads)
copy_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, size_t n16,
            const uint8_t* __restrict__ src_tail, uint8_t* __restrict__ dst_tail, int tail) {
  const size_t stride = static_cast<size_t>(gridDim.x) * kCopyThreads;
  size_t i = static_cast<size_t>(blockIdx.x) * kCopyThreads + threadIdx.x;
  // kCopyUnroll independent vectors in flight per thread
  for (; i + (kCopyUnroll - 1) * stride < n16; i += kCopyUnroll * stride) {
    uint4 v[kCopyUnroll];
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) v[u] = src[i + u * stride];
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) dst[i + u * stride] = v[u];
  }
  for (; i < n16; i += stride) dst[i] = src[i];
  if (blockIdx.x == 0 && static_cast<int>(threadIdx.x) < tail)
    dst_tail[threadIdx.x] = src_tail[threadIdx.x];
}

}  // namespace

cudaError_t launch_copy(const void* src, void* dst, size_t bytes, cudaStream_t stream) {
  const size_t n16 = bytes / 16;
  const int tail = static_cast<int>(bytes % 16);
  const size_t per_cta = static_cast<size_t>(kCopyThreads) * kCopyUnroll;
  size_t ctas = (n16 + per_cta - 1) / per_cta;
  if (ctas < 1) ctas = 1;
  if (ctas > static_cast<size_t>(kCopyMaxCtas)) ctas = kCopyMaxCtas;
  const uint8_t* s8 = static_cast<const uint8_t*>(src) + n16 * 16;
  uint8_t* d8 = static_cast<uint8_t*>(dst) + n16 * 16;
  copy_kernel<<<static_cast<unsigned>(ctas), kCopyThreads, 0, stream>>>(
      static_cast<const uint4*>(src), static_cast<uint4*>(dst), n16, s8, d8, tail);
  return cudaGetLastError();
}

}  // namespace zarya
