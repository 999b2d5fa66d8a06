// Reordering and restoration of Zarya's inference modes (Sec. 5.1 steps 2
// and 4, Sec. 5.2 steps 1 and 8) for sm_103a: one CTA per sequence.
//
// Reordering puts a sequence's unmasked positions first (in order) and its
// masked positions after them, in order or by ascending key (ties by
// position). A position's destination is its rank among the unmasked
// positions before it (a block-wide scan of ballots over 1024-position
// chunks), or n_unmasked plus its rank in the masked group: the number of
// masked positions before it, or, with keys, its place in the masked group
// sorted by (key, position): a bitonic sort of (key << 32 | position) in
// shared memory for rows up to kSortMax positions, else the number of masked
// positions with a smaller (key, position), counted against the keys staged
// in shared memory 1024 at a time. Restoration scatters through the
// permutation. Both move a few bytes per position: latency-bound.
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"
#include "token_ops.cuh"
#include "ptx.cuh"

namespace zarya {
namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int kSortMax = 4096;   // keyed rows up to this length are sorted in shared memory

// Exclusive rank of `flag` over the CTA's current chunk, plus the chunk's
// total; s_warp is kWarps ints of scratch.
__device__ __forceinline__ int block_rank(bool flag, int* s_warp, int& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned bal = __ballot_sync(0xffffffffu, flag);
  const int in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) s_warp[warp] = __popc(bal);
  __syncthreads();
  if (warp == 0) {
    const int v = s_warp[lane];
    int incl = v;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += o;
    }
    s_warp[lane] = incl - v;          // exclusive over warps
    if (lane == 31) s_warp[kWarps] = incl;
  }
  __syncthreads();
  const int r = s_warp[warp] + in_warp;
  total = s_warp[kWarps];
  __syncthreads();                    // s_warp is reused by the next call
  return r;
}

// Ascending bitonic sort of s[0, n2) (n2 a power of two) by the CTA.
__device__ __forceinline__ void bitonic_sort(uint64_t* s, int n2) {
  for (int k = 2; k <= n2; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < n2; i += kThreads) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const uint64_t x = s[i], y = s[ixj];
          const bool up = (i & k) == 0;
          if ((x > y) == up) {
            s[i] = y;
            s[ixj] = x;
          }
        }
      }
      __syncthreads();
    }
  }
}

__global__ void __launch_bounds__(kThreads) reorder_kernel(const ReorderParams a) {
  __shared__ int s_warp[kWarps + 1];
  __shared__ uint32_t s_key[kThreads];
  __shared__ uint8_t s_msk[kThreads];
  __shared__ uint64_t s_sort[kSortMax];   // keyed rows: (key << 32 | position) of the masked group
  grid_dependency_wait();
  grid_launch_dependents();
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  const int64_t base = static_cast<int64_t>(b) * a.max_len;
  int n = a.lens[b];
  if (n < 0 || n > a.max_len) {
    if (tid == 0) record_error(a.err, ZARYA_DEVERR_ROWS);
    n = 0;
  }
  const int32_t* tok = a.tokens + base;
  const uint8_t* msk = a.is_masked + base;
  const uint32_t* key = a.order_key != nullptr ? a.order_key + base : nullptr;
  int32_t* perm = a.perm + base;
  int32_t* out = a.tokens_out + base;

  // Unmasked count.
  int nvis = 0;
  for (int c0 = 0; c0 < n; c0 += kThreads) {
    const int i = c0 + tid;
    int total;
    block_rank(i < n && msk[i] == 0, s_warp, total);
    nvis += total;
  }
  // Destinations. Keyed rows up to kSortMax positions collect their masked
  // group in shared memory (in position order) and sort it below.
  const bool sort_keys = key != nullptr && n <= kSortMax;
  int vis_before = 0;
  for (int c0 = 0; c0 < n; c0 += kThreads) {
    const int i = c0 + tid;
    const bool in = i < n;
    const bool masked = in && msk[i] != 0;
    int total;
    const int r = block_rank(in && !masked, s_warp, total);
    int dest = -1;
    if (in) {
      const int masked_before = i - (vis_before + r);
      if (!masked) {
        dest = vis_before + r;
      } else if (key == nullptr) {
        dest = nvis + masked_before;
      } else if (sort_keys) {
        s_sort[masked_before] = (static_cast<uint64_t>(key[i]) << 32) | static_cast<uint32_t>(i);
      } else {
        dest = nvis;   // + the masked positions with a smaller (key, position), below
      }
    }
    if (key != nullptr && !sort_keys) {
      const uint32_t ki = masked ? key[i] : 0u;
      int smaller = 0;
      for (int j0 = 0; j0 < n; j0 += kThreads) {
        const int j = j0 + tid;
        s_key[tid] = j < n ? key[j] : 0u;
        s_msk[tid] = j < n ? msk[j] : 0;
        __syncthreads();
        if (masked) {
          const int m = min(kThreads, n - j0);
          for (int t = 0; t < m; ++t) {
            const uint32_t kj = s_key[t];
            const bool before = kj < ki || (kj == ki && j0 + t < i);
            smaller += (s_msk[t] != 0 && before) ? 1 : 0;
          }
        }
        __syncthreads();
      }
      if (masked) dest += smaller;
    }
    if (dest >= 0) {
      perm[dest] = i;
      out[dest] = tok[i];
    }
    vis_before += total;
  }
  if (sort_keys) {
    const int m = n - nvis;
    int n2 = 1;
    while (n2 < m) n2 <<= 1;
    for (int t = m + tid; t < n2; t += kThreads) s_sort[t] = ~0ull;
    __syncthreads();
    bitonic_sort(s_sort, n2);
    for (int t = tid; t < m; t += kThreads) {
      const int i = static_cast<int>(s_sort[t] & 0xffffffffu);
      perm[nvis + t] = i;
      out[nvis + t] = tok[i];
    }
  }
  // Positions past the sequence: no permutation entry, tokens as given.
  for (int i = n + tid; i < a.max_len; i += kThreads) {
    perm[i] = -1;
    out[i] = tok[i];
  }
  if (tid == 0) a.n_unmasked[b] = nvis;
}

__global__ void __launch_bounds__(kThreads) restore_kernel(const ReorderParams a) {
  grid_dependency_wait();
  grid_launch_dependents();
  const int b = blockIdx.x;
  const int64_t base = static_cast<int64_t>(b) * a.max_len;
  int n = a.lens[b];
  if (n < 0 || n > a.max_len) {
    if (threadIdx.x == 0) record_error(a.err, ZARYA_DEVERR_ROWS);
    n = 0;
  }
  const int32_t* tok = a.tokens + base;
  const int32_t* perm = a.perm_in + base;
  int32_t* out = a.tokens_out + base;
  for (int i = threadIdx.x; i < n; i += kThreads) {
    const int p = perm[i];
    if (p < 0 || p >= n) record_error(a.err, ZARYA_DEVERR_PERM);
    else out[p] = tok[i];
  }
  for (int i = n + threadIdx.x; i < a.max_len; i += kThreads) out[i] = tok[i];
}

}  // namespace

cudaError_t launch_reorder(const ReorderParams& p, cudaStream_t stream) {
  PdlLaunch l(dim3(static_cast<unsigned>(p.B)), dim3(kThreads), 0, stream);
  return cudaLaunchKernelEx(&l.cfg, reorder_kernel, p);
}

cudaError_t launch_restore(const ReorderParams& p, cudaStream_t stream) {
  PdlLaunch l(dim3(static_cast<unsigned>(p.B)), dim3(kThreads), 0, stream);
  return cudaLaunchKernelEx(&l.cfg, restore_kernel, p);
}

}  // namespace zarya
