// Repetition penalty over logits rows (Sec. 5.1 step 3 and Table 2: the
// per-step draws honour temperature, top_p and repetition_penalty) for
// sm_103a, in place: every token that occurs in its sequence's history has
// its logit multiplied by the penalty when negative and divided by it
// otherwise, once per distinct token however often it occurs.
//
// One CTA per logits row: it finds the row's sequence (binary search over the
// dense row layout), marks the history's tokens in a shared-memory bitmap of
// the vocabulary (an atomic OR per occurrence, so duplicates collapse), then
// rewrites the marked logits in float32, rounding back to bf16 to nearest
// even for bf16 rows. Latency-bound: a few thousand tokens per row.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"
#include "token_ops.cuh"
#include "ptx.cuh"

namespace zarya {
namespace {

constexpr int kPenaltyThreads = 256;

__device__ __forceinline__ float penalized(float x, float p) { return x < 0.f ? x * p : x / p; }

__global__ void __launch_bounds__(kPenaltyThreads) penalty_kernel(const PenaltyParams a) {
  extern __shared__ uint32_t bitmap[];
  __shared__ int s_seq;
  grid_dependency_wait();
  grid_launch_dependents();
  const int g = blockIdx.x;
  const int tid = threadIdx.x;
  if (tid == 0) {
    // the sequence b with row_offsets[b] <= g < row_offsets[b + 1], or -1
    int lo = 0, hi = a.B - 1, b = -1;
    while (lo <= hi) {
      const int mid = (lo + hi) >> 1;
      if (a.row_offsets[mid] <= g) {
        b = mid;
        lo = mid + 1;
      } else {
        hi = mid - 1;
      }
    }
    if (b >= 0 && g >= a.row_offsets[b + 1]) b = -1;
    s_seq = b;
  }
  const int nwords = (a.V + 31) >> 5;
  for (int w = tid; w < nwords; w += kPenaltyThreads) bitmap[w] = 0u;
  __syncthreads();
  const int b = s_seq;
  if (b < 0) return;   // a row of no sequence: left as it is
  const int h0 = a.hist_offsets[b], h1 = a.hist_offsets[b + 1];
  if (h0 < 0 || h1 < h0 || h1 > a.n_hist) {
    if (tid == 0) record_error(a.err, ZARYA_DEVERR_ROWS);
    return;
  }
  for (int i = h0 + tid; i < h1; i += kPenaltyThreads) {
    const int tok = a.hist_tokens[i];
    if (tok < 0 || tok >= a.V) {
      record_error(a.err, ZARYA_DEVERR_TOKEN);
      continue;
    }
    atomicOr(&bitmap[tok >> 5], 1u << (tok & 31));
  }
  __syncthreads();
  const int64_t base = static_cast<int64_t>(g) * a.row_stride;
  for (int w = tid; w < nwords; w += kPenaltyThreads) {
    uint32_t bits = bitmap[w];
    while (bits != 0u) {
      const int v = (w << 5) + __ffs(bits) - 1;
      bits &= bits - 1u;
      if (a.bf16) {
        __nv_bfloat16* x = static_cast<__nv_bfloat16*>(a.logits) + base + v;
        *x = __float2bfloat16_rn(penalized(__bfloat162float(*x), a.penalty));
      } else {
        float* x = static_cast<float*>(a.logits) + base + v;
        *x = penalized(*x, a.penalty);
      }
    }
  }
}

}  // namespace

cudaError_t launch_penalty(const PenaltyParams& p, cudaStream_t stream) {
  const size_t smem = static_cast<size_t>((p.V + 31) >> 5) * sizeof(uint32_t);
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(penalty_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  PdlLaunch l(dim3(static_cast<unsigned>(p.rows)), dim3(kPenaltyThreads), smem, stream);
  return cudaLaunchKernelEx(&l.cfg, penalty_kernel, p);
}

}  // namespace zarya
