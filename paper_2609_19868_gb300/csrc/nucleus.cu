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
// The masses differ from exact ones by the fp32 exponent argument's rounding
// (below 1e-6 relative for any token within 2^20 of the maximum's mass), the
// approximate exp2 (2^-22) and the truncation to 2^-40 (masses below that count
// as zero): a kept set can differ from the exact one only where the mass at
// its boundary lies within about 1e-6 of top_p. Each lane adds into its own slot
// of each bin (no two lanes of a warp share a word). The row is read, in
// 16-byte vectors, once for its maximum, once per digit and once for the
// masking writes.
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
// One histogram per CTA with a private slot per lane: bin b, lane l at
// hist[b * kHistStride + l]. No two lanes of a warp ever add to the same
// word (a warp's adds never serialise on an address, whatever the digits),
// and the padding slot makes the per-bin sums below bank-conflict free.
constexpr int kHistStride = 33;
constexpr size_t kNucSmem = 256 * kHistStride * sizeof(unsigned long long);

__device__ __forceinline__ float nuc_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// floor(e * 2^40) for e in [0, 1] (the mass in 2^-40 fixed point), from the
// float's fields: e = mant * 2^(ex - 23) with the implicit bit in mant.
// NaN (never a mass of a finite logit) counts as 0.
__device__ __forceinline__ unsigned long long mass_fixed(float e) {
  const uint32_t u = __float_as_uint(e);
  const int sh = static_cast<int>(u >> 23) - 127 + 40 - 23;
  if (sh > 17 || sh <= -24) return 0ull;   // NaN / above 1, or below 2^-40
  const unsigned long long mant = (u & 0x7FFFFFu) | 0x800000u;
  return sh >= 0 ? (mant << sh) : (mant >> (-sh));
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

// The logits of 16-byte vector w.
template <typename TBits>
struct Vec16 {
  static constexpr int kN = 16 / sizeof(TBits);
  TBits e[kN];
  __device__ __forceinline__ explicit Vec16(const uint4& w) {
    const TBits* p = reinterpret_cast<const TBits*>(&w);
#pragma unroll
    for (int k = 0; k < kN; ++k) e[k] = p[k];
  }
};

template <typename TBits>
__global__ void __launch_bounds__(kNucThreads) nucleus_kernel(const NucleusParams a) {
  constexpr int kKeyBits = 8 * static_cast<int>(sizeof(TBits));
  constexpr int kPerVec = 16 / static_cast<int>(sizeof(TBits));
  extern __shared__ unsigned long long hist[];   // [256][kHistStride]
  __shared__ unsigned long long bins[256];
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
  // the row as 16-byte vectors (rows start 16-byte aligned), then a scalar tail
  const uint4* row4 = reinterpret_cast<const uint4*>(row);
  const int nvec = V / kPerVec;
  const int tail0 = nvec * kPerVec;

  // the row's maximum
  float m = -INFINITY;
  for (int i = tid; i < nvec; i += kNucThreads) {
    const Vec16<TBits> w(row4[i]);
#pragma unroll
    for (int k = 0; k < kPerVec; ++k) m = fmaxf(m, bits_to_float(w.e[k]));
  }
  for (int v = tail0 + tid; v < V; v += kNucThreads) m = fmaxf(m, bits_to_float(row[v]));
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
    for (int i = tid; i < 256 * kHistStride; i += kNucThreads) hist[i] = 0ull;
    __syncthreads();
    auto add = [&](TBits b) {
      const uint32_t key = logit_key(b);
      if (level > 0 && (key >> (shift + 8)) != prefix) return;
      const unsigned long long q = mass_fixed(nuc_ex2(fmaf(bits_to_float(b), a.k2, neg_mk)));
      if (q != 0ull) atomicAdd(&hist[((key >> shift) & 255u) * kHistStride + lane], q);
    };
    for (int i = tid; i < nvec; i += kNucThreads) {
      const Vec16<TBits> w(row4[i]);
#pragma unroll
      for (int k = 0; k < kPerVec; ++k) add(w.e[k]);
    }
    for (int v = tail0 + tid; v < V; v += kNucThreads) add(row[v]);
    __syncthreads();
    if (tid < 256) {
      unsigned long long t = 0;
#pragma unroll 8
      for (int l = 0; l < 32; ++l) t += hist[tid * kHistStride + l];
      bins[tid] = t;
    }
    __syncthreads();
    if (tid == 0) {
      if (level == 0) {
        unsigned long long tot = 0;
        for (int b = 0; b < 256; ++b) tot += bins[b];
        s_total = tot;
      }
      const double target = static_cast<double>(a.top_p) * static_cast<double>(s_total);
      unsigned long long cum = above;
      int pick = -1, lowest = -1;
      for (int b = 255; b >= 0; --b) {
        const unsigned long long h = bins[b];
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
        for (int b = 255; b > pick; --b) cum += bins[b];
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
  uint4* wrow4 = reinterpret_cast<uint4*>(row);
  for (int i = tid; i < nvec; i += kNucThreads) {
    uint4 w = wrow4[i];
    TBits* e = reinterpret_cast<TBits*>(&w);
    bool cut = false;
#pragma unroll
    for (int k = 0; k < kPerVec; ++k)
      if (logit_key(e[k]) < prefix) {
        e[k] = neg_inf;
        cut = true;
      }
    if (cut) wrow4[i] = w;
  }
  for (int v = tail0 + tid; v < V; v += kNucThreads)
    if (logit_key(row[v]) < prefix) row[v] = neg_inf;
}

}  // namespace

cudaError_t launch_nucleus(const NucleusParams& p, cudaStream_t stream) {
  // the histogram's dynamic shared memory is above the default 48 KB limit
  constexpr int kMaxDevices = 64;
  static int configured[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  if (!__atomic_load_n(&configured[dev], __ATOMIC_ACQUIRE)) {
    e = cudaFuncSetAttribute(nucleus_kernel<uint16_t>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kNucSmem));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(nucleus_kernel<uint32_t>,
                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(kNucSmem));
    if (e != cudaSuccess) return e;
    __atomic_store_n(&configured[dev], 1, __ATOMIC_RELEASE);
  }
  PdlLaunch l(dim3(static_cast<unsigned>(p.rows)), dim3(kNucThreads), kNucSmem, stream);
  if (p.bf16) return cudaLaunchKernelEx(&l.cfg, nucleus_kernel<uint16_t>, p);
  return cudaLaunchKernelEx(&l.cfg, nucleus_kernel<uint32_t>, p);
}

}  // namespace zarya
