// zarya_slot_attn_noalloc: slot attention whose split-KV scratch lives in a
// fixed, library-owned device array instead of a caller-provided workspace.
//
// Some callers cannot allocate device memory when they run attention: a
// serving engine that has already handed all of HBM to its own KV-cache pool,
// a host application that forbids its plug-ins from allocating device memory,
// or a latency-critical decode loop that cannot afford cudaMalloc/cudaFree
// (both may synchronise the device). For them this entry point takes the same
// inputs and outputs as zarya_slot_attn but no workspace, and allocates
// nothing: the scratch is a file-scope __device__ array of kScratchBytes that
// every GPU which loads the library keeps until the process exits.
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"

namespace zarya {
namespace {

constexpr size_t kScratchBytes = size_t(16) << 20;  // 16 MiB per device

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// Device address of g_noalloc_scratch on the current device. In host code the
// symbol itself is only a host-side stand-in; the real address comes from
// cudaGetSymbolAddress, looked up once per device and cached.
void* scratch_address(cudaError_t* status) {
  constexpr int kMaxDevices = 64;
  static void* cache[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    *status = (e != cudaSuccess) ? e : cudaErrorInvalidDevice;
    return nullptr;
  }
  void* ptr = __atomic_load_n(&cache[dev], __ATOMIC_ACQUIRE);
  if (ptr == nullptr) {
    e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess || ptr == nullptr) {
      *status = (e != cudaSuccess) ? e : cudaErrorInvalidSymbol;
      return nullptr;
    }
    __atomic_store_n(&cache[dev], ptr, __ATOMIC_RELEASE);
  }
  *status = cudaSuccess;
  return ptr;
}

}  // namespace
}  // namespace zarya

extern "C" {

zarya_status zarya_slot_attn_noalloc(const void* q, const void* k_cache, const void* v_cache,
                                     const int32_t* cache_lens, const int32_t* page_table,
                                     const int32_t* n_slots, const int32_t* slot_len,
                                     const int32_t* mask_mode, void* out,
                                     const zarya_attn_desc* desc, zarya_stream_t stream_) {
  if (desc == nullptr || q == nullptr) return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  // Make the stream's device current: the scratch address and the split plan
  // (which depends on the SM count) are per device.
  cudaError_t ce = zarya::select_device(stream, q);
  if (ce != cudaSuccess) return zarya::cuda_fail("selecting the stream's device", ce);

  const size_t need = zarya_slot_attn_workspace_size(desc);
  if (need > zarya::kScratchBytes) return ZARYA_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  if (need > 0) {
    scratch = zarya::scratch_address(&ce);
    if (scratch == nullptr) return zarya::cuda_fail("looking up the scratch address", ce);
    // The split counters, when the plan has them, sit at the end of the
    // workspace layout and must start at zero; the array keeps whatever the
    // last call left. (A dispatch order needs no clearing: it is rewritten
    // by every call.)
    const size_t cnt_bytes = zarya::workspace_counter_bytes(desc);
    if (cnt_bytes > need)
      return zarya::cuda_fail("split counter layout does not fit the scratch plan",
                              cudaErrorInvalidValue);
    if (cnt_bytes > 0) {
      ce = cudaMemsetAsync(static_cast<unsigned char*>(scratch) + (need - cnt_bytes), 0,
                           cnt_bytes, stream);
      if (ce != cudaSuccess) return zarya::cuda_fail("clearing the split counters", ce);
    }
  }
  return zarya_slot_attn(q, k_cache, v_cache, cache_lens, page_table, n_slots, slot_len,
                         mask_mode, out, scratch, need > 0 ? zarya::kScratchBytes : 0, desc,
                         stream_);
}

}  // extern "C"
