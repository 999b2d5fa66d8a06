// top_p (nucleus) truncation of logits rows (Sec. 5.1 step 3 and Table 2: the
// per-step draws honour temperature, top_p and repetition_penalty) for
// sm_103a, in place: the logits of a row below its threshold x* become -inf,
// where x* is the largest logit value whose tokens, with every token above
// it, hold at least top_p of the row's probability softmax(x / T). The draws
// that follow then run over the nucleus with renormalised probabilities.
//
// One CTA per row. x* is found by radix descent over the order-preserving
// integer key of the logit (sign-flipped bits; 16 bits for bf16, 32 for
// fp32), 8 bits per pass: a pass adds each qualifying element's mass
// exp((x - m) / T) to a 256-bin histogram of its next key digit, and the bin
// where the mass counted from the top reaches top_p of the total fixes that
// digit. Masses are summed in 2^-40 fixed point (64-bit integers), so the sums,
// and with them the boundary, do not depend on the order of the atomics.
// The row is read once for its maximum, once per digit and once for the
// masking writes: latency- and L2-bound, small beside the draws.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "internal.cuh"
#include "token_ops.cuh"
#include "ptx.cuh"

namespace zarya {
namespace {

constexpr int kNucThreads = 512;
constexpr int kNucWarps = kNucThreads / 32;

__device__ __forceinline__ float nuc_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Order-preserving key of a logit and the logit of a key.
__device__ __forceinline__ uint32_t logit_key(uint16_t b) {
  return b ^ ((b & 0x8000u) ? 0xFFFFu : 0x8000u);
}
__device__ __forceinline__ uint32_t logit_key(uint32_t b) {
  return b ^ ((b & 0x80000000u) ? 0xFFFFFFFFu : 0x80000000u);
}

template <typename TBits>
__device__ __forceinline__ float bits_to_float(TBits b) {
  if (sizeof(TBits) == 2) return __uint_as_float(static_cast<uint32_t>(b) << 16);
  return __uint_as_float(static_cast<uint32_t>(b));
}

template <typename TBits>
__global__ void __launch_bounds__(kNucThreads) nucleus_kernel(const NucleusParams a) {
  constexpr int kKeyBits = 8 * static_cast<int>(sizeof(TBits));
  __shared__ unsigned long long hist[kNucWarps][256];
  __shared__ float s_max[kNucWarps];
  __shared__ uint32_t s_prefix;
  __shared__ unsigned long long s_above, s_total;
  grid_dependency_wait();
  grid_launch_dependents();
  const int g = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  if (g < a.row_offsets[0] || g >= a.row_offsets[a.B]) return;   // a row of no sequence
  TBits* row = static_cast<TBits*>(a.logits) + static_cast<int64_t>(g) * a.row_stride;
  const int V = a.V;

  // the row's maximum
  float m = -INFINITY;
  for (int v = tid; v < V; v += kNucThreads) m = fmaxf(m, bits_to_float(row[v]));
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, d));
  if (lane == 0) s_max[warp] = m;
  __syncthreads();
  m = s_max[0];
  for (int w = 1; w < kNucWarps; ++w) m = fmaxf(m, s_max[w]);
  if (!(m > -INFINITY)) return;   // every logit -inf (or NaN): nothing to cut

  const float neg_mk = -m * a.k2;
  uint32_t prefix = 0;
  unsigned long long above = 0;   // mass of the keys above the current prefix's range
  for (int level = 0; level < kKeyBits / 8; ++level) {
    const int shift = kKeyBits - 8 * (level + 1);
    for (int i = tid; i < kNucWarps * 256; i += kNucThreads) (&hist[0][0])[i] = 0ull;
    __syncthreads();
    for (int v = tid; v < V; v += kNucThreads) {
      const TBits b = row[v];
      const uint32_t key = logit_key(b);
      if (level > 0 && (key >> (shift + 8)) != prefix) continue;
      const float e = nuc_ex2(fmaf(bits_to_float(b), a.k2, neg_mk));
      const unsigned long long q = __float2ull_rz(e * 0x1p40f);
      if (q != 0ull) atomicAdd(&hist[warp][(key >> shift) & 255u], q);
    }
    __syncthreads();
    if (tid < 256) {
      unsigned long long t = 0;
      for (int w = 0; w < kNucWarps; ++w) t += hist[w][tid];
      hist[0][tid] = t;
    }
    __syncthreads();
    if (tid == 0) {
      if (level == 0) {
        unsigned long long tot = 0;
        for (int b = 0; b < 256; ++b) tot += hist[0][b];
        s_total = tot;
      }
      const double target = static_cast<double>(a.top_p) * static_cast<double>(s_total);
      unsigned long long cum = above;
      int pick = -1, lowest = -1;
      for (int b = 255; b >= 0; --b) {
        const unsigned long long h = hist[0][b];
        if (h == 0ull) continue;
        lowest = b;
        if (static_cast<double>(cum + h) >= target) {
          pick = b;
          break;
        }
        cum += h;
      }
      if (pick < 0) {   // the target is beyond the mass (rounding): keep down to the lowest bin
        pick = lowest < 0 ? 0 : lowest;
        cum = above;
        for (int b = 255; b > pick; --b) cum += hist[0][b];
      }
      s_prefix = (prefix << 8) | static_cast<uint32_t>(pick);
      s_above = cum;
    }
    __syncthreads();
    prefix = s_prefix;
    above = s_above;
    __syncthreads();   // hist is cleared by the next level
  }
  // prefix is now the key of x*: every logit below it becomes -inf
  const TBits neg_inf = sizeof(TBits) == 2 ? static_cast<TBits>(0xFF80u)
                                           : static_cast<TBits>(0xFF800000u);
  for (int v = tid; v < V; v += kNucThreads)
    if (logit_key(row[v]) < prefix) row[v] = neg_inf;
}

}  // namespace

cudaError_t launch_nucleus(const NucleusParams& p, cudaStream_t stream) {
  PdlLaunch l(dim3(static_cast<unsigned>(p.rows)), dim3(kNucThreads), 0, stream);
  if (p.bf16) return cudaLaunchKernelEx(&l.cfg, nucleus_kernel<uint16_t>, p);
  return cudaLaunchKernelEx(&l.cfg, nucleus_kernel<uint32_t>, p);
}

}  // namespace zarya
