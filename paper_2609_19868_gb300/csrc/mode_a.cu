// Mode A mask-budget planning (Sec. 5.1 step 1) for sm_103a: one CTA per
// sequence. Every binomial draw is the sum of Bernoulli trials [u < p] over
// Philox4x32-10 uniforms (counter (trial / 4, sequence, draw, offset), word
// trial % 4): the CTA's threads take four trials per Philox block and a
// block-wide sum gives the count. Draw 0 is the diffusion total
// Binomial(n, alpha_0); draw 1 + s is diffusion step s, Binomial(remaining,
// 1 / (T - s)); the tokens left after the T diffusion steps are revealed one
// per step. With T = 0, ceil(n / 4) steps of 4. Latency-bound (a block
// reduction per diffusion step).
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"
#include "token_ops.cuh"
#include "philox.cuh"
#include "ptx.cuh"

namespace zarya {
namespace {

constexpr int kThreads = 256;

// Number of trials i < n (of this sequence's draw) with u_i < p.
__device__ __forceinline__ int bernoulli_count(const ModeAParams& a, int b, int draw, int n,
                                               float p, int* s_red) {
  int c = 0;
  for (int q = threadIdx.x; 4 * q < n; q += kThreads) {
    const uint4 w = philox4x32_10(make_uint4(static_cast<uint32_t>(q), static_cast<uint32_t>(b),
                                             static_cast<uint32_t>(draw), a.ctr3),
                                  a.key0, a.key1);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (4 * q + j < n && uniform_from_word(ws[j]) < p) ++c;
  }
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) c += __shfl_xor_sync(0xffffffffu, c, d);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) s_red[warp] = c;
  __syncthreads();
  int total = 0;
#pragma unroll
  for (int w = 0; w < kThreads / 32; ++w) total += s_red[w];
  __syncthreads();
  return total;
}

__global__ void __launch_bounds__(kThreads) mode_a_budget_kernel(const ModeAParams a) {
  __shared__ int s_red[kThreads / 32];
  grid_dependency_wait();
  grid_launch_dependents();
  const int b = blockIdx.x;
  int32_t* row = a.counts + static_cast<int64_t>(b) * a.max_steps;
  const int n = a.n_masked[b];
  int steps = 0;
  bool ok = n >= 0;
  if (ok && n > 0) {
    if (a.T <= 0) {
      steps = (n + 3) / 4;
      ok = steps <= a.max_steps;
      if (ok)
        for (int s = threadIdx.x; s < steps; s += kThreads)
          row[s] = s < steps - 1 ? 4 : n - 4 * (steps - 1);
    } else {
      const int n_diff = bernoulli_count(a, b, 0, n, a.alpha0, s_red);
      steps = a.T + (n - n_diff);
      ok = static_cast<long long>(a.T) + (n - n_diff) <= a.max_steps;
      if (ok) {
        int remaining = n_diff;
        for (int s = 0; s < a.T; ++s) {
          const float p = 1.0f / static_cast<float>(a.T - s);
          const int k = bernoulli_count(a, b, 1 + s, remaining, p, s_red);
          if (threadIdx.x == 0) row[s] = k;
          remaining -= k;
        }
        for (int s = a.T + threadIdx.x; s < steps; s += kThreads) row[s] = 1;
      }
    }
  }
  if (!ok) {
    if (threadIdx.x == 0) record_error(a.err, ZARYA_DEVERR_ROWS);
    steps = 0;
  }
  for (int s = steps + threadIdx.x; s < a.max_steps; s += kThreads) row[s] = 0;
  if (threadIdx.x == 0) a.n_steps[b] = steps;
}

}  // namespace

cudaError_t launch_mode_a_budget(const ModeAParams& p, cudaStream_t stream) {
  PdlLaunch l(dim3(static_cast<unsigned>(p.B)), dim3(kThreads), 0, stream);
  return cudaLaunchKernelEx(&l.cfg, mode_a_budget_kernel, p);
}

}  // namespace zarya
