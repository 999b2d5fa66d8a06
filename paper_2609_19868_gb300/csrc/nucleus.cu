// top_p (nucleus) truncation of logits rows (Sec. 5.1 step 3 and Table 2: the
// per-step draws honour temperature, top_p and repetition_penalty) for
// sm_103a, in place: the logits of a row below its threshold x* become -inf,
// where x* is the largest logit value whose tokens, with every token above
// it, hold at least top_p of the row's probability softmax(x / T). The draws
// that follow then run over the nucleus with renormalised probabilities.
//
// One CTA per row, no atomics. With a = (x - m) log2(e) / T (one fused
// multiply-add, monotone in x; m the row's maximum) a token's mass relative
// to the maximum's is 2^a. Stage 1 sorts the tokens into one-octave mass
// bins, j = floor(-a) for a in (-42, 0] (lighter tokens count as massless);
// since j falls as x grows, each bin holds a contiguous range of logit
// values. Every thread adds its tokens' masses into private slots, the slots
// are summed in a fixed order, and the bin where the mass counted from the
// top reaches top_p of the total contains x*. One warp then finds that bin's
// range of order-preserving logit keys (sign-flipped bits; 16 bits for bf16,
// 32 for fp32) by a 32-way search over the monotone bin function, a pass over
// the row gathers the keys in that range into shared memory (each warp its
// own segment, placed by a warp prefix sum of the lanes' counts), and stage 2
// runs a radix descent over them, 4 bits of the key offset per level, again
// with private slots per thread: a level sums each candidate's mass into its
// digit, and the digit where the mass counted from the top reaches top_p is
// fixed. A row whose bin holds more keys than the shared memory takes the
// descent's levels over the row instead. The last pass cuts every logit
// below x* (a float comparison, so a signed zero equal to x* stays, and NaN
// logits are left in place).
//
// Masses are fixed point relative to their bin: a token of bin j adds
// floor(2^(a + j + 22)) (between 2^21 and 2^22) in units of 2^-(j + 22), and
// the decisions compare integer sums in one unit (2^-42 of the maximum's mass;
// the target ceil(top_p x total) exactly), so the boundary does not depend on
// the order of the GPU's additions (a thread's slots hold at most 1023
// tokens, so 32 bits never overflow). The masses
// differ from exact ones by the fp32 exponent argument's rounding (below 1e-6
// relative for any token within 2^20 of the maximum's mass), the approximate
// exp2 (2^-22) and the truncation (below 2^-21 relative; tokens under 2^-42 of
// the maximum count as zero): a kept set can differ from the exact one only
// where the mass at its boundary lies within about 1e-6 of top_p. The row is
// read, in 16-byte vectors with several in flight per thread, once for its
// maximum, once for the mass bins, once to gather the candidates and once for
// the masking writes; after the first read it sits in L2.
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
constexpr int kNucUnroll = 4;   // 16-byte loads in flight per thread
// Mass bins: bin j holds the tokens with a in (-j - 1, -j].
constexpr int kMassBins = 42;
constexpr float kMassFloor = -42.f;
constexpr float kMassFloorUp = -41.999996185302734375f;   // the float just above -42
// floor(-c) for c in [-42, 0] from the bits of fma_rz(c, -1, 1.5 * 2^23)
constexpr float kBinMagic = 12582912.f;
constexpr uint32_t kBinMagicBits = 0x4B400000u;
// The descent's digits: 4 bits of the key offset per level.
constexpr int kDigitBits = 4;
constexpr int kDigits = 1 << kDigitBits;
// Shared memory: stage 1's private slots (bin j, thread t at j * kNucThreads
// + t, 32 bits); afterwards the descent's private slots (digit k, thread t at
// k * kNucThreads + t) and, behind them, the candidates' keys, one segment of
// kCandBytes / kNucWarps bytes per warp.
constexpr size_t kNucSmem = static_cast<size_t>(kMassBins) * kNucThreads * sizeof(uint32_t);
constexpr size_t kDigitBytes = static_cast<size_t>(kDigits) * kNucThreads * sizeof(uint32_t);
constexpr size_t kCandBytes = kNucSmem - kDigitBytes;
// A bin of at most this many keys counts its gathered keys per key (32-bit
// counts in the digit area, beside the candidates) and scans the counts for
// x* instead of descending over the digits.
constexpr int kHistKeys = 4096;
static_assert(kHistKeys * sizeof(uint32_t) <= kDigitBytes, "the key counts sit in the digit area");
// A thread adds at most this many tokens into a 32-bit slot (each at most
// 2^22 + 1): up to ceil(V / (kPerVec * kNucThreads)) vectors of kPerVec and
// one tail token, which kNucleusMaxVocab keeps within it.
constexpr int kMaxTokensPerThread = 1023;
static_assert(((kNucleusMaxVocab / 8 + kNucThreads - 1) / kNucThreads) * 8 + 1 <= kMaxTokensPerThread &&
                  ((kNucleusMaxVocab / 4 + kNucThreads - 1) / kNucThreads) * 4 + 1 <= kMaxTokensPerThread,
              "a thread's 32-bit mass slots could overflow");
static_assert(static_cast<unsigned long long>(kMaxTokensPerThread) * ((1u << 22) + 1u) < (1ull << 32),
              "a thread's 32-bit mass slots could overflow");

__device__ __forceinline__ float nuc_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// The decisions compare masses in one fixed-point unit, 2^-42 of the
// maximum's mass (bin 20's unit): bin j's integer sums scaled by 2^(20 - j),
// the lighter bins' shifted right (each losing less than one unit). The
// row's total stays below 2^61 (V < 2^19 tokens of at most 2^42 units).
constexpr int kCommonBin = 20;
__device__ __forceinline__ unsigned long long to_common(unsigned long long t, int j) {
  return j <= kCommonBin ? (t << (kCommonBin - j)) : (t >> (j - kCommonBin));
}

// ceil(t p) for p in (0, 1) and t < 2^61, exactly: p's 24-bit significand
// times t in 128 bits, shifted right by p's binary exponent, rounded up.
__device__ __forceinline__ unsigned long long mul_frac_ceil(unsigned long long t, float p) {
  const uint32_t u = __float_as_uint(p);
  const int ex = static_cast<int>((u >> 23) & 0xFFu);
  const unsigned long long mant = (u & 0x7FFFFFu) | (ex != 0 ? 0x800000u : 0u);
  const int shift = 150 - (ex != 0 ? ex : 1);   // p = mant 2^-shift, shift >= 24
  const unsigned long long lo = t * mant, hi = __umul64hi(t, mant);
  unsigned long long q, rem;
  if (shift >= 128) {
    q = 0;
    rem = lo | hi;
  } else if (shift >= 64) {
    q = hi >> (shift - 64);
    rem = lo | (hi & ((1ull << (shift - 64)) - 1ull));
  } else {
    q = (lo >> shift) | (hi << (64 - shift));
    rem = lo & ((1ull << shift) - 1ull);
  }
  return q + (rem != 0ull ? 1ull : 0ull);
}

// A token's mass in its bin's units, and its bin. The same arithmetic decides
// the bins in stage 1, in the key-range search and in stage 2. The mass is
// floor(e 2^(j + 22)) for e = 2^c: the product is exact (a power of two), and
// adding 2^23 with rounding toward zero leaves floor(v) in the low bits (v is
// below 2^23), so the sum's bits minus 2^23's are the integer mass.
struct Mass {
  uint32_t q;   // 0 for a massless token (a <= -42, or NaN)
  uint32_t j;
};
// The exponent argument a = (x - m) k2: the difference and the product each
// round within 2^-24 of their own value, so a is within 2^-23 |a| of exact
// (the heavy tokens near a = 0 nearly exact); x k2 - m k2 would carry the
// rounding of m k2, up to 2^-25 |m k2| whatever a is, into every token's
// argument and lift the tokens nearest the maximum above 0. It is monotone
// in x, so each bin is a range of keys.
__device__ __forceinline__ float mass_arg(float x, float m, float k2) {
  return __fmul_rn(__fsub_rn(x, m), k2);
}

__device__ __forceinline__ Mass token_mass(float x, float k2, float m) {
  const float a = mass_arg(x, m, k2);
  const float c = a > kMassFloor ? fminf(a, 0.f) : -INFINITY;   // -inf: e = 0
  const uint32_t j =
      __float_as_uint(__fmaf_rz(fmaxf(c, kMassFloorUp), -1.f, kBinMagic)) - kBinMagicBits;
  const float scale = __uint_as_float((j + 149u) << 23);   // 2^(j + 22)
  const float v = nuc_ex2(c) * scale;
  return Mass{__float_as_uint(__fadd_rz(v, 8388608.f)) - 0x4B000000u, j};
}

// token_mass for two logits at once: the same operations, the ones with a
// paired fp32 form taken two at a time (each half rounds exactly as the
// scalar instruction does), so each result is token_mass's bit for bit.
__device__ __forceinline__ void token_mass2(float x0, float x1, float k2, float m, Mass& s0,
                                            Mass& s1) {
  const float2 a = __fmul2_rn(__fadd2_rn(make_float2(x0, x1), make_float2(-m, -m)), make_float2(k2, k2));
  // a <= 0 for every token of the row (x <= m): token_mass's clamp at 0 is
  // the identity here (a signed zero gives the same bin and mass either way)
  const float c0 = a.x > kMassFloor ? a.x : -INFINITY;
  const float c1 = a.y > kMassFloor ? a.y : -INFINITY;
  const float2 y = __ffma2_rz(make_float2(fmaxf(c0, kMassFloorUp), fmaxf(c1, kMassFloorUp)),
                              make_float2(-1.f, -1.f), make_float2(kBinMagic, kBinMagic));
  s0.j = __float_as_uint(y.x) - kBinMagicBits;
  s1.j = __float_as_uint(y.y) - kBinMagicBits;
  const float2 scale = make_float2(__uint_as_float((s0.j + 149u) << 23),
                                   __uint_as_float((s1.j + 149u) << 23));
  const float2 v = __fmul2_rn(make_float2(nuc_ex2(c0), nuc_ex2(c1)), scale);
  const float2 r = __fadd2_rz(v, make_float2(8388608.f, 8388608.f));
  s0.q = __float_as_uint(r.x) - 0x4B000000u;
  s1.q = __float_as_uint(r.y) - 0x4B000000u;
}

// The bin of a logit (kMassBins for a massless one): token_mass's bin test.
__device__ __forceinline__ int token_bin(float x, float k2, float m) {
  const float a = mass_arg(x, m, k2);
  if (!(a > kMassFloor)) return kMassBins;
  const float c = fminf(fmaxf(a, kMassFloorUp), 0.f);
  return static_cast<int>(__float_as_uint(__fmaf_rz(c, -1.f, kBinMagic)) - kBinMagicBits);
}

// Order-preserving key of a logit given as fp32 bits (bf16 logits widened),
// kKeyBits wide, and the fp32 bits of a key.
template <int kKeyBits>
__device__ __forceinline__ uint32_t logit_key(uint32_t f) {
  const uint32_t k = f ^ (static_cast<uint32_t>(static_cast<int32_t>(f) >> 31) | 0x80000000u);
  return k >> (32 - kKeyBits);
}
template <int kKeyBits>
__device__ __forceinline__ uint32_t key_bits(uint32_t key) {
  const uint32_t k = key << (32 - kKeyBits);
  return (k & 0x80000000u) ? (k ^ 0x80000000u) : ~k & (0xFFFFFFFFu << (32 - kKeyBits));
}

// Calls f(fp32 bits, fp32 bits) for each pair of logits of a 16-byte vector.
template <typename TBits, typename F>
__device__ __forceinline__ void each_logit_pair(const uint4& v, F&& f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if (sizeof(TBits) == 2) {
#pragma unroll
    for (int k = 0; k < 4; ++k) f(w[k] << 16, w[k] & 0xFFFF0000u);
  } else {
    f(w[0], w[1]);
    f(w[2], w[3]);
  }
}

// Calls f(fp32 bits) for each logit of a 16-byte vector.
template <typename TBits, typename F>
__device__ __forceinline__ void each_logit(const uint4& v, F&& f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    if (sizeof(TBits) == 2) {
      f(w[k] << 16);
      f(w[k] & 0xFFFF0000u);
    } else {
      f(w[k]);
    }
  }
}

template <typename TBits>
__device__ __forceinline__ uint32_t widen(TBits b) {
  return sizeof(TBits) == 2 ? static_cast<uint32_t>(b) << 16 : static_cast<uint32_t>(b);
}

// Calls f(w, i) on this thread's 16-byte vectors i = tid, tid + kNucThreads,
// ... of v[0, n), with kNucUnroll loads in flight before the first is used.
template <typename F>
__device__ __forceinline__ void for_each_vec(const uint4* v, int n, int tid, F&& f) {
  int i = tid;
  for (; i + (kNucUnroll - 1) * kNucThreads < n; i += kNucUnroll * kNucThreads) {
    uint4 w[kNucUnroll];
#pragma unroll
    for (int u = 0; u < kNucUnroll; ++u) w[u] = v[i + u * kNucThreads];
#pragma unroll
    for (int u = 0; u < kNucUnroll; ++u) f(w[u], i + u * kNucThreads);
  }
  for (; i < n; i += kNucThreads) f(v[i], i);
}

// The smallest key in [lo, hi] whose pred holds, hi + 1 if none; pred is
// monotone (false ... false true ... true). Called by one whole warp; every
// lane returns the same key.
template <typename P>
__device__ __forceinline__ uint32_t first_true_key(uint32_t lo, uint32_t hi, int lane, P&& pred) {
  uint64_t a = lo, b = static_cast<uint64_t>(hi) + 1;   // the answer lies in [a, b]
  while (a < b) {
    const uint64_t step = (b - a + 31) >> 5;
    const uint64_t probe = a + static_cast<uint64_t>(lane) * step;
    const bool p = probe < b && pred(static_cast<uint32_t>(probe));
    const unsigned bal = __ballot_sync(0xffffffffu, p);
    const int last = 31 - __clz(__ballot_sync(0xffffffffu, probe < b));   // the last lane with a probe
    const int f = bal ? __ffs(bal) - 1 : last + 1;   // the first lane whose probe holds
    if (f == 0) return static_cast<uint32_t>(a);
    const uint64_t na = a + static_cast<uint64_t>(f - 1) * step + 1;
    b = f <= last ? a + static_cast<uint64_t>(f) * step : b;
    a = na;
  }
  return static_cast<uint32_t>(a);
}

template <typename TBits>
__global__ void __launch_bounds__(kNucThreads, 2) nucleus_kernel(const NucleusParams a) {
  constexpr int kKeyBits = 8 * static_cast<int>(sizeof(TBits));
  constexpr int kPerVec = 16 / static_cast<int>(sizeof(TBits));
  constexpr int kSegKeys = static_cast<int>(kCandBytes / sizeof(TBits)) / kNucWarps;
  extern __shared__ __align__(16) uint32_t smem[];
  __shared__ unsigned long long bins[kMassBins];
  __shared__ float s_max[kNucWarps];
  __shared__ int s_seg[kNucWarps];
  __shared__ int s_pick, s_over;
  __shared__ uint32_t s_klo, s_khi, s_prefix;
  __shared__ unsigned long long s_above, s_target;
  __shared__ unsigned long long s_wsum[kNucWarps];
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

  // the row's maximum (NaN ignored)
  float m = -INFINITY;
  if constexpr (sizeof(TBits) == 2) {
    __nv_bfloat162 m2 = __float2bfloat162_rn(-INFINITY);
    for_each_vec(row4, nvec, tid, [&](const uint4& v, int) {
      const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
      m2 = __hmax2(m2, __hmax2(__hmax2(h[0], h[1]), __hmax2(h[2], h[3])));
    });
    m = fmaxf(__low2float(m2), __high2float(m2));
  } else {
    for_each_vec(row4, nvec, tid, [&](const uint4& v, int) {
      m = fmaxf(m, fmaxf(fmaxf(__uint_as_float(v.x), __uint_as_float(v.y)),
                         fmaxf(__uint_as_float(v.z), __uint_as_float(v.w))));
    });
  }
  for (int v = tail0 + tid; v < V; v += kNucThreads) m = fmaxf(m, __uint_as_float(widen(row[v])));
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, d));
  if (lane == 0) s_max[warp] = m;
  __syncthreads();
  m = s_max[0];
  for (int w = 1; w < kNucWarps; ++w) m = fmaxf(m, s_max[w]);
  if (!(m > -INFINITY)) return;   // every logit -inf (or NaN): nothing to cut
  const float k2 = a.k2;

  // Stage 1: the mass bins in private slots. A slot has one writer, so its
  // updates are shared-memory reductions (no load-add-store chain from one
  // logit to the next, and integer sums do not depend on their order).
  uint32_t* own = smem + tid;
#pragma unroll
  for (int j = 0; j < kMassBins; ++j) own[j * kNucThreads] = 0u;
  auto add_mass2 = [&](uint32_t f0, uint32_t f1) {
    Mass s0, s1;
    token_mass2(__uint_as_float(f0), __uint_as_float(f1), k2, m, s0, s1);
    atomicAdd(own + s0.j * kNucThreads, s0.q);
    atomicAdd(own + s1.j * kNucThreads, s1.q);
  };
  for_each_vec(row4, nvec, tid, [&](const uint4& v, int) { each_logit_pair<TBits>(v, add_mass2); });
  for (int v = tail0 + tid; v < V; v += kNucThreads) {
    const Mass s = token_mass(__uint_as_float(widen(row[v])), k2, m);
    atomicAdd(own + s.j * kNucThreads, s.q);
  }
  __syncthreads();
  for (int j = warp; j < kMassBins; j += kNucWarps) {   // fixed summation order
    unsigned long long t = 0;
    for (int i = lane; i < kNucThreads; i += 32) t += smem[j * kNucThreads + i];
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) t += __shfl_xor_sync(0xffffffffu, t, d);
    if (lane == 0) bins[j] = t;
  }
  __syncthreads();
  if (tid == 0) {
    unsigned long long tot = 0;
#pragma unroll 1
    for (int j = 0; j < kMassBins; ++j) tot += to_common(bins[j], j);
    const unsigned long long target = tot > 0 ? mul_frac_ceil(tot, a.top_p) : 0ull;
    int pick = -1, lowest = -1;
    unsigned long long cum = 0;
    if (tot > 0) {
#pragma unroll 1
      for (int j = 0; j < kMassBins; ++j) {
        if (bins[j] == 0ull) continue;
        const unsigned long long h = to_common(bins[j], j);
        lowest = j;
        if (cum + h >= target) {
          pick = j;
          break;
        }
        cum += h;
      }
      if (pick < 0) {   // the target is beyond the mass (truncation): keep down to the lowest bin
        pick = lowest;
        cum = 0;
#pragma unroll 1
        for (int j = 0; j < pick; ++j) cum += to_common(bins[j], j);
      }
    }
    s_pick = pick;
    s_above = cum;
    s_target = target;
    s_over = 0;
  }
  __syncthreads();
  const int jbin = s_pick;
  if (jbin < 0) return;   // no token has mass (a +inf logit): nothing to cut

  // The key range of bin jbin (the bin falls as the key grows; NaN keys lie
  // outside [key(-inf), key(+inf)]), cut at the maximum: no token lies above
  // it, and bin 0 would otherwise reach to +inf (one past the maximum's key,
  // so that +0 stays inside when the maximum came out as -0).
  if (warp == 0) {
    const uint32_t lo = logit_key<kKeyBits>(0xFF800000u), hi = logit_key<kKeyBits>(0x7F800000u);
    auto bin_of = [&](uint32_t key) {
      return token_bin(__uint_as_float(key_bits<kKeyBits>(key)), k2, m);
    };
    const uint32_t klo = first_true_key(lo, hi, lane, [&](uint32_t k) { return bin_of(k) <= jbin; });
    const uint32_t kend = first_true_key(lo, hi, lane, [&](uint32_t k) { return bin_of(k) < jbin; });
    if (lane == 0) {
      s_klo = klo;
      s_khi = min(kend - 1, logit_key<kKeyBits>(__float_as_uint(m)) + 1u);
    }
  }
  __syncthreads();
  const uint32_t klo = s_klo, range = s_khi - s_klo;
  uint32_t prefix = 0;   // the key offset of x* above the current level
  if (range > 0) {
    // Each lane marks its logits in [x(klo), x(khi)] (a float test that takes
    // every key of the range; a signed zero it takes beside them fails the
    // key test that follows) in a bit mask per vector.
    const uint32_t flo = key_bits<kKeyBits>(klo), fhi = key_bits<kKeyBits>(s_khi);
    // bit e set: logit e of the vector is in the range
    auto in_bits = [&](const uint4& v) -> uint32_t {
      if constexpr (sizeof(TBits) == 2) {
        const uint32_t lo2 = (flo >> 16) | (flo & 0xFFFF0000u), hi2 = (fhi >> 16) | (fhi & 0xFFFF0000u);
        const __nv_bfloat162 lo = *reinterpret_cast<const __nv_bfloat162*>(&lo2);
        const __nv_bfloat162 hi = *reinterpret_cast<const __nv_bfloat162*>(&hi2);
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
        uint32_t x = 0;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          x |= ((__hge2_mask(h[k], lo) & __hle2_mask(h[k], hi)) & 0x00010001u) << (2 * k);
        return (x | (x >> 15)) & 0xFFu;
      } else {
        const float lo = __uint_as_float(flo), hi = __uint_as_float(fhi);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
        uint32_t x = 0;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float f = __uint_as_float(w[k]);
          x |= static_cast<uint32_t>(f >= lo && f <= hi) << k;
        }
        return x;
      }
    };
    // the fp32 bits of logit e of a vector
    auto logit_bits = [&](const uint4& v, int e) -> uint32_t {
      const int k = sizeof(TBits) == 2 ? e >> 1 : e;   // the 32-bit word (selects, no local array)
      const uint32_t x = k < 2 ? (k == 0 ? v.x : v.y) : (k == 2 ? v.z : v.w);
      if constexpr (sizeof(TBits) == 2) {
        return (e & 1) ? (x & 0xFFFF0000u) : (x << 16);
      } else {
        return x;
      }
    };
    const bool narrow = range < static_cast<uint32_t>(kHistKeys);   // unsigned: an fp32 bin can span 2^31 keys
    uint32_t* hist = smem;   // a narrow bin's count per key (the digit area)
    if (narrow) {
      for (int i = tid; i <= static_cast<int>(range); i += kNucThreads) hist[i] = 0u;
      if (tid == 0) s_prefix = 0xFFFFFFFFu;
    }
    // Gather the keys of the bin into this warp's segment: a warp prefix sum
    // of the lanes' counts places them. The loop runs the same number of times
    // in every lane of the warp (the shuffles need all 32).
    TBits* seg = reinterpret_cast<TBits*>(reinterpret_cast<unsigned char*>(smem) + kDigitBytes) +
                 warp * kSegKeys;
    int cnt = 0;   // keys this warp found (uniform over the warp)
    const int warp0 = tid - lane;
    for (int i0 = warp0; i0 < nvec; i0 += kNucUnroll * kNucThreads) {
      uint4 w[kNucUnroll];
      uint32_t bits[kNucUnroll];
      int c = 0;
#pragma unroll
      for (int u = 0; u < kNucUnroll; ++u) {
        const int i = i0 + u * kNucThreads + lane;
        w[u] = i < nvec ? row4[i] : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < kNucUnroll; ++u) {
        bits[u] = i0 + u * kNucThreads + lane < nvec ? in_bits(w[u]) : 0u;
        c += __popc(bits[u]);
      }
      int incl = c;   // inclusive prefix sum of the lanes' counts
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int t = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += t;
      }
      int pos = cnt + incl - c;
#pragma unroll
      for (int u = 0; u < kNucUnroll; ++u) {
        for (uint32_t mb = bits[u]; mb != 0u; mb &= mb - 1u, ++pos) {
          const int e = __ffs(mb) - 1;
          if (pos < kSegKeys) seg[pos] = static_cast<TBits>(logit_key<kKeyBits>(logit_bits(w[u], e)));
        }
      }
      cnt += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (warp == 0) {   // the scalar tail (fewer than kPerVec logits)
      const bool valid = tail0 + lane < V;
      const uint32_t key = valid ? logit_key<kKeyBits>(widen(row[tail0 + lane])) : 0u;
      const bool in = valid && key - klo <= range;
      const unsigned bal = __ballot_sync(0xffffffffu, in);
      const int p = cnt + __popc(bal & ((1u << lane) - 1u));
      if (in && p < kSegKeys) seg[p] = static_cast<TBits>(key);
      cnt += __popc(bal);
    }
    if (lane == 0) {
      s_seg[warp] = min(cnt, kSegKeys);
      if (cnt > kSegKeys) s_over = 1;
    }
    __syncthreads();
    const bool over = s_over != 0;
    const int n_mine = s_seg[warp];

    if (narrow) {
      // Stage 2, narrow bin: how many tokens hold each key of the bin (the
      // tokens of one key share its logit and so its mass), counted over the
      // gathered keys (over the row when a segment overflowed), then x* by a
      // scan from the largest key down, each key's mass its count times the
      // mass of its logit: the same integer sums as adding the tokens one by
      // one. A lane holds the last key it met with its count so far and adds
      // them when another key comes (or at the end): a row where one key holds
      // most of the bin's tokens then makes few atomics on that key.
      uint32_t run_key = 0xFFFFFFFFu, run_cnt = 0u;
      auto count_d = [&](uint32_t d) {
        if (d > range) return;
        if (d != run_key) {
          if (run_cnt != 0u) atomicAdd(hist + run_key, run_cnt);
          run_key = d;
          run_cnt = 0u;
        }
        ++run_cnt;
      };
      if (!over) {
        for (int e = lane; e < n_mine; e += 32) count_d(static_cast<uint32_t>(seg[e]) - klo);
      } else {
        for_each_vec(row4, nvec, tid, [&](const uint4& v, int) {
          for (uint32_t b = in_bits(v); b != 0u; b &= b - 1u)
            count_d(logit_key<kKeyBits>(logit_bits(v, __ffs(b) - 1)) - klo);
        });
        for (int v = tail0 + tid; v < V; v += kNucThreads) count_d(logit_key<kKeyBits>(widen(row[v])) - klo);
      }
      if (run_cnt != 0u) atomicAdd(hist + run_key, run_cnt);
      __syncthreads();
      const int nk = static_cast<int>(range) + 1;
      // key r from the top (r = 0 is key klo + range): its mass in the common unit
      auto key_mass = [&](int r) -> unsigned long long {
        const uint32_t c = hist[range - r];
        if (c == 0u) return 0ull;
        const uint32_t key = klo + range - static_cast<uint32_t>(r);
        const uint32_t q = token_mass(__uint_as_float(key_bits<kKeyBits>(key)), k2, m).q;
        return to_common(static_cast<unsigned long long>(c) * q, jbin);
      };
      // Thread t takes the keys r in [t c, (t + 1) c): their mass, a block
      // prefix sum over the threads in order, and the one thread whose keys
      // hold the crossing of the target walks them.
      const int chunk = (nk + kNucThreads - 1) / kNucThreads;
      const int r0 = min(tid * chunk, nk), r1 = min(r0 + chunk, nk);
      unsigned long long mine = 0;
      for (int r = r0; r < r1; ++r) mine += key_mass(r);
      unsigned long long incl = mine;
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const unsigned long long t = __shfl_up_sync(0xffffffffu, incl, d);
        if (lane >= d) incl += t;
      }
      if (lane == 31) s_wsum[warp] = incl;
      __syncthreads();
      const unsigned long long target = s_target;
      unsigned long long cum = s_above + (incl - mine);   // mass above this thread's first key
      for (int w = 0; w < warp; ++w) cum += s_wsum[w];
      if (cum < target && target <= cum + mine) {
        for (int r = r0; r < r1; ++r) {
          const unsigned long long h = key_mass(r);
          if (cum + h >= target) {
            s_prefix = range - static_cast<uint32_t>(r);
            break;
          }
          cum += h;
        }
      }
      __syncthreads();
      const bool beyond = s_prefix == 0xFFFFFFFFu;   // the same in every thread
      __syncthreads();
      if (beyond) {   // the target is beyond the mass (truncation): keep down to the lowest key with mass
        for (int r = r1 - 1; r >= r0; --r) {
          if (hist[range - r] != 0u) {
            atomicMin(&s_prefix, range - static_cast<uint32_t>(r));
            break;
          }
        }
        __syncthreads();
      }
      prefix = s_prefix == 0xFFFFFFFFu ? 0u : s_prefix;
    } else {
      // Stage 2, wide bin: the radix descent over d = key - klo, kDigitBits per
      // level, over the gathered keys (or the row, when a segment overflowed).
      const int nbits = 32 - __clz(range);
      const int levels = (nbits + kDigitBits - 1) / kDigitBits;
      const unsigned long long target = s_target;
      unsigned long long above = s_above;   // mass of the tokens above the current range
      for (int level = 0; level < levels; ++level) {
        const int shift = kDigitBits * (levels - 1 - level);
#pragma unroll
        for (int k = 0; k < kDigits; ++k) own[k * kNucThreads] = 0u;
        auto add = [&](uint32_t key) {
          const uint32_t d = key - klo;
          if (d > range) return;
          if (level > 0 && (d >> (shift + kDigitBits)) != prefix) return;
          const Mass s = token_mass(__uint_as_float(key_bits<kKeyBits>(key)), k2, m);
          atomicAdd(own + ((d >> shift) & (kDigits - 1)) * kNucThreads, s.q);
        };
        if (!over) {
          for (int e = lane; e < n_mine; e += 32) add(seg[e]);
        } else {
          for_each_vec(row4, nvec, tid, [&](const uint4& v, int) {
            each_logit<TBits>(v, [&](uint32_t f) { add(logit_key<kKeyBits>(f)); });
          });
          for (int v = tail0 + tid; v < V; v += kNucThreads) add(logit_key<kKeyBits>(widen(row[v])));
        }
        __syncthreads();
        if (warp < kDigits) {   // digit `warp`'s total, in a fixed order
          unsigned long long t = 0;
          for (int i = lane; i < kNucThreads; i += 32) t += smem[warp * kNucThreads + i];
#pragma unroll
          for (int d = 16; d >= 1; d >>= 1) t += __shfl_xor_sync(0xffffffffu, t, d);
          if (lane == 0) bins[warp] = t;
        }
        __syncthreads();
        if (tid == 0) {
          unsigned long long cum = above;
          int pick = -1, lowest = -1;
#pragma unroll 1
          for (int k = kDigits - 1; k >= 0; --k) {
            if (bins[k] == 0ull) continue;
            const unsigned long long h = to_common(bins[k], jbin);
            lowest = k;
            if (cum + h >= target) {
              pick = k;
              break;
            }
            cum += h;
          }
          if (pick < 0) {   // the target is beyond the mass (truncation): keep down to the lowest digit
            pick = lowest < 0 ? 0 : lowest;
            cum = above;
#pragma unroll 1
            for (int k = kDigits - 1; k > pick; --k) cum += to_common(bins[k], jbin);
          }
          s_prefix = (prefix << kDigitBits) | static_cast<uint32_t>(pick);
          s_above = cum;
        }
        __syncthreads();
        prefix = s_prefix;
        above = s_above;
      }
    }
  }

  // x* is the logit of key klo + prefix: every logit below it becomes -inf
  // (a float comparison: a signed zero equal to x* is kept, and NaN logits
  // stay in place)
  const uint32_t xbits = key_bits<kKeyBits>(klo + prefix);
  uint4* wrow4 = reinterpret_cast<uint4*>(row);
  if constexpr (sizeof(TBits) == 2) {
    const uint32_t x2 = (xbits >> 16) | (xbits & 0xFFFF0000u);
    const __nv_bfloat162 xs = *reinterpret_cast<const __nv_bfloat162*>(&x2);
    for_each_vec(row4, nvec, tid, [&](const uint4& v, int i) {
      uint32_t w[4] = {v.x, v.y, v.z, v.w};
      uint32_t any = 0;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t cut = __hlt2_mask(*reinterpret_cast<const __nv_bfloat162*>(&w[k]), xs);
        w[k] = (w[k] & ~cut) | (0xFF80FF80u & cut);
        any |= cut;
      }
      if (any) wrow4[i] = make_uint4(w[0], w[1], w[2], w[3]);
    });
  } else {
    const float xs = __uint_as_float(xbits);
    for_each_vec(row4, nvec, tid, [&](const uint4& v, int i) {
      uint32_t w[4] = {v.x, v.y, v.z, v.w};
      bool any = false;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const bool cut = __uint_as_float(w[k]) < xs;
        w[k] = cut ? 0xFF800000u : w[k];
        any = any || cut;
      }
      if (any) wrow4[i] = make_uint4(w[0], w[1], w[2], w[3]);
    });
  }
  const TBits neg_inf = sizeof(TBits) == 2 ? static_cast<TBits>(0xFF80u)
                                           : static_cast<TBits>(0xFF800000u);
  for (int v = tail0 + tid; v < V; v += kNucThreads)
    if (__uint_as_float(widen(row[v])) < __uint_as_float(xbits)) row[v] = neg_inf;
}

}  // namespace

cudaError_t launch_nucleus(const NucleusParams& p, cudaStream_t stream) {
  // the private slots' dynamic shared memory is above the default 48 KB limit
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
