// Slot selection and token acceptance of Zarya's slotted speculative decoding
// (Sec. 5.2 steps 3-6) for sm_103a.
//
// Row pass (one CTA per logits row): streams the row's V logits once with
// 16-byte non-allocating loads and reduces, in fp32, the row maximum m, the
// sum s of 2^((x - m) * log2(e) / T), and
//   - the draft form at T = 0: the first index of the maximum (step 3);
//   - the draft form at T > 0: the first index of the maximum of
//     x / T + g_v, with the Gumbel noise g_v generated in registers from
//     Philox4x32-10 (step 4);
//   - the verification form: the logit of the row's given token (step 6).
// Probability of the drawn / given token t: 2^((x_t - m) * log2(e) / T) / s.
// The pass reads V * element-size bytes per row and writes 8: HBM-bound at
// T = 0, bound by the integer and special-function work of the noise at
// T > 0.
//
// Sequence pass: the draft form (one CTA, since the verification layout is a
// running sum over the batch) selects the slots (step 5) and lays out the
// verification block; the verification form (one warp per sequence) scans the
// accepted prefixes (step 6).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstring>
#include <cstdint>

#include "internal.cuh"
#include "token_ops.cuh"
#include "philox.cuh"
#include "ptx.cuh"

namespace zarya {
namespace {

// Row pass: a producer warp streams the row into a ring of shared-memory
// stages with bulk copies; kConsumerWarps warps reduce the staged vectors.
constexpr int kConsumerWarps = 8;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kRowThreads = kConsumers + 32;
constexpr int kStages = 4;
constexpr int kChunkVecs = 1024;                 // 16-byte vectors per stage (16 KB)
constexpr int kVecsPerThread = kChunkVecs / kConsumers;
constexpr size_t kRowSmemBytes = static_cast<size_t>(kStages) * kChunkVecs * 16;
constexpr int kRowCtasPerSm = 3;
constexpr uint64_t kWaitNs = 2000000000ull;     // 2 s: a stage that never fills
constexpr int kSelectThreads = 1024;
constexpr int kAcceptThreads = 256;
constexpr float kLog2e = 1.4426950408889634f;

enum RowMode { kDraftArgmax = 0, kDraftGumbel = 1, kVerify = 2 };

struct RowArgs {
  const void* logits;
  int64_t row_stride;       // elements
  const int32_t* row_offsets;
  const int32_t* tokens;    // verification: token of every row
  int32_t* out_token;       // draft: drawn token of every row
  float* out_prob;          // probability of the drawn / given token
  int* err;
  int B, V, total_rows;
  float inv_t;              // 1 / T (1 at T = 0)
  float k2;                 // log2(e) / T (log2(e) at T = 0)
  uint32_t key0, key1;      // Philox key
  uint32_t ctr2, ctr3;      // Philox counter words 2 and 3 (the offset)
  int parts;                // CTAs per row: a thread-block cluster when > 1
};

// Bulk copy of `bytes` (a multiple of 16, both ends 16-byte aligned) from
// global memory into this CTA's shared memory; completes as transaction bytes
// on the mbarrier `bar`.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes,
                                          uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float bf16_bits_to_f32(uint32_t b) { return __uint_as_float(b << 16); }

__device__ __forceinline__ __nv_bfloat162 as_bf162(uint32_t w) {
  __nv_bfloat162 r;
  memcpy(&r, &w, sizeof r);
  return r;
}

// Standard Gumbel variate from a uniform u in (0, 1] (see uniform_from_word):
// E = -log1p(-u) exponential, g = -log(E); g decreases as u grows.
__device__ __forceinline__ float gumbel_from_uniform(float u) {
  const float e = -log1pf(-u);
  return -__logf(e);
}

__device__ __forceinline__ float gumbel_from_word(uint32_t w) {
  return gumbel_from_uniform(uniform_from_word(w));
}

// Per-thread reduction state of the row pass.
struct RowState {
  float m;     // running maximum of x
  float s;     // sum of 2^((x - m) k2) over the elements seen
  float bz;    // Gumbel: best x / T + g
  float bx;    // Gumbel: x at the best index
  int bi;      // first index of the best value (INT_MAX: none yet)
};

// Exponent (x - m) * k2 as one fused multiply-add against -m * k2: a single
// rounding of the exact difference, and the rounding of m * k2 is common to
// every term of the row (it cancels in the probability).
__device__ __forceinline__ float lg_term(float x, float k2, float neg_mk) {
  return fmaf(x, k2, neg_mk);
}

// New running maximum vm > st.m: rescale the sum to it.
__device__ __forceinline__ void absorb_max(RowState& st, float vm, float k2) {
  const float neg_mk = -vm * k2;
  st.s = st.s * ex2(lg_term(st.m, k2, neg_mk));  // st.m = -inf gives 0 * 0
  st.m = vm;
}

// Upper bound of any Gumbel variate gumbel_from_word makes: the smallest u is
// 2^-33, where E = -log1p(-u) is 2^-33 to within float rounding and
// g = -log(E) = 33 ln 2 = 22.87; 24 leaves room for the approximate log.
constexpr float kGumbelMax = 24.0f;

// Floats ordered as ints (for atomicMax on shared memory): non-negative
// floats keep their bits, negative ones flip all bits but the sign.
__device__ __forceinline__ int float_order(float f) {
  const int b = __float_as_int(f);
  return b >= 0 ? b : b ^ 0x7fffffff;
}
__device__ __forceinline__ float order_float(int k) {
  return __int_as_float(k >= 0 ? k : k ^ 0x7fffffff);
}

// Gumbel selection over one vector of the row (its softmax terms are added
// by absorb_chunk). `bound` (or the thread's own best, if larger) is a score
// x / T + g that some element of the row reaches: a vector whose largest
// possible score, fma(max x, 1/T, kGumbelMax), stays below it cannot hold the
// draw and skips its noise. Otherwise an element reaches the threshold only
// if its noise exceeds t = thr - max x / T (less 0.01 for the rounding of the
// noise and of the score), i.e. only if E = -log1p(-u) < exp(-t), i.e. only if
// u < u_lim = -expm1(-exp(-t)). Since u_lim <= exp(-t), the words are cut at
// the larger exp(-t + 0.001) (one ex2; the 0.001 covers its rounding): a word
// above the cut has u > u_lim and skips both logarithms, and the elements let
// through beyond u_lim score below the threshold, so the draw is the same.
// Every element that reaches the test gets its exact score.
template <int kN>
__device__ __forceinline__ void gumbel_select(RowState& st, const float (&x)[kN], int v0,
                                              const RowArgs& a, uint32_t row, float bound) {
  float vm = x[0];
#pragma unroll
  for (int j = 1; j < kN; ++j) vm = fmaxf(vm, x[j]);
  const float thr = fmaxf(bound, st.bz);
  if (fmaf(vm, a.inv_t, kGumbelMax) < thr) return;
  uint32_t w_cut = 0xffffffffu;
  if (thr > -INFINITY) {
    const float t = thr - vm * a.inv_t - 0.011f;
    const float lim = ex2(-t * kLog2e);
    // u(w) >= w 2^-32 (1 - 2^-23) for every word w, so u(w) <= lim only if
    // w <= lim 2^32 (1 + 2^-22); the float product below rounds to no less.
    if (lim < 1.f) {
      const float c = lim * 0x1p32f * (1.f + 0x1p-21f);
      w_cut = c >= 0x1p32f ? 0xffffffffu : static_cast<uint32_t>(c);
    }
  }
  // kN is 4 or 8 with v0 a multiple of 4: one Philox block per 4 elements.
#pragma unroll
  for (int q = 0; q < kN / 4; ++q) {
    const uint32_t blk = static_cast<uint32_t>((v0 >> 2) + q);
    const uint4 w = philox4x32_10(make_uint4(blk, row, a.ctr2, a.ctr3), a.key0, a.key1);
    const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (ws[j] > w_cut) continue;
      const float z = fmaf(x[q * 4 + j], a.inv_t, gumbel_from_uniform(uniform_from_word(ws[j])));
      const int v = v0 + q * 4 + j;
      if (z > st.bz || (z == st.bz && v < st.bi)) {
        st.bz = z;
        st.bi = v;
        st.bx = x[q * 4 + j];
      }
    }
  }
}

// The draft (T = 0) and verification forms over one stage: thread t's
// kVecsPerThread vectors of the chunk, x[k] holding elements e0 + k * estride
// .. e0 + k * estride + kN - 1 (vectors past the row hold -inf). One maximum
// and one rescale test per chunk, and independent partial sums.
template <int kMode, int kN>
__device__ __forceinline__ void absorb_chunk(RowState& st, const float (&x)[kVecsPerThread][kN],
                                             float vm, int e0, int estride, float k2) {
  if (vm > st.m) {
    if (kMode == kDraftArgmax) {
      int best = 0x7fffffff;
#pragma unroll
      for (int k = kVecsPerThread - 1; k >= 0; --k)
#pragma unroll
        for (int j = kN - 1; j >= 0; --j)
          if (x[k][j] == vm) best = e0 + k * estride + j;
      st.bi = best;
    }
    absorb_max(st, vm, k2);
  }
  if (st.m > -INFINITY) {
    const float neg_mk = -st.m * k2;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int k = 0; k < kVecsPerThread; ++k)
#pragma unroll
      for (int j = 0; j < kN; ++j) acc[j & 3] += ex2(lg_term(x[k][j], k2, neg_mk));
    st.s += (acc[0] + acc[1]) + (acc[2] + acc[3]);
  }
}

// One scalar element at index v (the row's ragged tail).
template <int kMode>
__device__ __forceinline__ void absorb_one(RowState& st, float x, int v, const RowArgs& a,
                                           uint32_t row) {
  if (x > st.m) {
    if (kMode == kDraftArgmax) st.bi = v;
    absorb_max(st, x, a.k2);
  }
  if (st.m > -INFINITY) st.s += ex2(lg_term(x, a.k2, -st.m * a.k2));
  if (kMode == kDraftGumbel) {
    const uint4 w = philox4x32_10(make_uint4(static_cast<uint32_t>(v >> 2), row, a.ctr2, a.ctr3),
                                  a.key0, a.key1);
    const int j = v & 3;
    const uint32_t wj = j == 0 ? w.x : (j == 1 ? w.y : (j == 2 ? w.z : w.w));
    const float z = fmaf(x, a.inv_t, gumbel_from_word(wj));
    if (z > st.bz || (z == st.bz && v < st.bi)) {
      st.bz = z;
      st.bi = v;
      st.bx = x;
    }
  }
}

// Merges state o into st (o covers other indices of the same row).
template <int kMode>
__device__ __forceinline__ void merge(RowState& st, const RowState& o, float k2) {
  const float mn = fmaxf(st.m, o.m);
  if (mn > -INFINITY) {
    const float neg_mk = -mn * k2;
    // A sum already relative to the maximum keeps its scale exactly.
    const float a = st.m == mn ? st.s : (st.m > -INFINITY ? st.s * ex2(lg_term(st.m, k2, neg_mk)) : 0.f);
    const float b = o.m == mn ? o.s : (o.m > -INFINITY ? o.s * ex2(lg_term(o.m, k2, neg_mk)) : 0.f);
    st.s = a + b;
  }
  if (kMode == kDraftArgmax) {
    if (o.m > st.m || (o.m == st.m && o.bi < st.bi)) st.bi = o.bi;
  } else if (kMode == kDraftGumbel) {
    if (o.bz > st.bz || (o.bz == st.bz && o.bi < st.bi)) {
      st.bz = o.bz;
      st.bi = o.bi;
      st.bx = o.bx;
    }
  }
  st.m = mn;
}

template <int kMode>
__device__ __forceinline__ RowState shfl_state(const RowState& st, int delta) {
  RowState o;
  o.m = __shfl_xor_sync(0xffffffffu, st.m, delta);
  o.s = __shfl_xor_sync(0xffffffffu, st.s, delta);
  o.bi = __shfl_xor_sync(0xffffffffu, st.bi, delta);
  if (kMode == kDraftGumbel) {
    o.bz = __shfl_xor_sync(0xffffffffu, st.bz, delta);
    o.bx = __shfl_xor_sync(0xffffffffu, st.bx, delta);
  } else {
    o.bz = o.bx = 0.f;
  }
  return o;
}

__device__ __forceinline__ void reset(RowState& st) {
  st.m = -INFINITY;
  st.s = 0.f;
  st.bz = -INFINITY;
  st.bx = 0.f;
  st.bi = 0x7fffffff;
}

template <typename TIn>
__device__ __forceinline__ void widen(const uint4& v, float (&x)[16 / sizeof(TIn)]) {
  if (sizeof(TIn) == 2) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      x[2 * j] = bf16_bits_to_f32(w[j] & 0xffffu);
      x[2 * j + 1] = __uint_as_float(w[j] & 0xffff0000u);
    }
  } else {
    x[0] = __uint_as_float(v.x);
    x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z);
    x[3] = __uint_as_float(v.w);
  }
}

// Maximum of a thread's vectors of one stage: bf16 pairs compared packed
// (the maximum of bf16 values is exact in either form), fp32 elementwise.
template <typename TIn>
__device__ __forceinline__ float chunk_max(const uint4 (&v)[kVecsPerThread],
                                           const float (&x)[kVecsPerThread][16 / sizeof(TIn)]) {
  if (sizeof(TIn) == 2) {
    __nv_bfloat162 m2 = as_bf162(v[0].x);
#pragma unroll
    for (int k = 0; k < kVecsPerThread; ++k) {
      if (k > 0) m2 = __hmax2(m2, as_bf162(v[k].x));
      m2 = __hmax2(m2, as_bf162(v[k].y));
      m2 = __hmax2(m2, as_bf162(v[k].z));
      m2 = __hmax2(m2, as_bf162(v[k].w));
    }
    return fmaxf(__low2float(m2), __high2float(m2));
  } else {
    float m = x[0][0];
#pragma unroll
    for (int k = 0; k < kVecsPerThread; ++k)
#pragma unroll
      for (int j = 0; j < 16 / static_cast<int>(sizeof(TIn)); ++j) m = fmaxf(m, x[k][j]);
    return m;
  }
}

// Row pass. With a.parts > 1 the CTAs of a row form a thread-block cluster:
// rank r streams the r-th contiguous share of the row's 16-byte vectors (the
// last rank also the ragged tail), and rank 0 merges the ranks' states
// through distributed shared memory.
//
// Within a CTA, warp kConsumerWarps (one lane) is the producer: it fills a
// ring of kStages shared-memory stages of kChunkVecs vectors with bulk copies
// (full[s] completes on the copy's bytes) and refills a stage once every
// consumer warp has released it (empty[s]). The consumer warps read each
// stage with 16-byte shared loads, thread t taking vectors t, t + 256, ...,
// so every thread sees its elements in increasing index order (the first
// maximum is kept by strict comparisons). Every wait is bounded; a timeout
// sets the error word and the CTA drains its copies before it leaves.
template <typename TIn, int kMode>
__global__ void __launch_bounds__(kRowThreads, kRowCtasPerSm) row_pass_kernel(const RowArgs a) {
  extern __shared__ __align__(128) uint4 stage_buf[];
  __shared__ uint64_t full[kStages], empty[kStages];
  __shared__ int best_score;   // Gumbel form: the CTA's best score so far (float_order)
  __shared__ RowState red[kConsumerWarps];
  __shared__ RowState cta_state;
  __shared__ int abort_flag;
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int st = 0; st < kStages; ++st) {
      mbar_init(&full[st], 1);
      mbar_init(&empty[st], kConsumerWarps);
    }
    abort_flag = 0;
    best_score = float_order(-INFINITY);
    fence_mbar_init();
  }
  __syncthreads();
  grid_dependency_wait();
  grid_launch_dependents();
  const int parts = a.parts;
  const int g = static_cast<int>(blockIdx.x) / parts;
  const int rank = parts > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int lo = a.row_offsets[0];
  const int hi = min(a.row_offsets[a.B], a.total_rows);
  if (g < lo || g >= hi) return;  // the whole cluster leaves together

  constexpr int kEpv = 16 / static_cast<int>(sizeof(TIn));  // elements per 16-byte vector
  const TIn* row = static_cast<const TIn*>(a.logits) + static_cast<int64_t>(g) * a.row_stride;
  const int nvec = a.V / kEpv;
  const int share = (nvec + parts - 1) / parts;
  const int v_lo = min(nvec, rank * share);
  const int v_hi = min(nvec, v_lo + share);
  const int nchunks = (v_hi - v_lo + kChunkVecs - 1) / kChunkVecs;
  const uint4* rowv = reinterpret_cast<const uint4*>(row) + v_lo;

  RowState st;
  reset(st);
  float x_tok = 0.f;
  bool tok_ok = true;

  if (warp == kConsumerWarps) {
    // Producer.
    if (lane == 0) {
      int issued = 0;
      for (int c = 0; c < nchunks; ++c) {
        const int sidx = c % kStages;
        if (c >= kStages &&
            !mbar_wait(&empty[sidx], ((c / kStages) - 1) & 1, kWaitNs, &abort_flag))
          break;
        if (*static_cast<volatile int*>(&abort_flag)) break;
        const int nv = min(kChunkVecs, v_hi - v_lo - c * kChunkVecs);
        const uint32_t bytes = static_cast<uint32_t>(nv) * 16u;
        mbar_arrive_expect_tx(&full[sidx], bytes);
        bulk_load(smem_u32(stage_buf + sidx * kChunkVecs), rowv + c * kChunkVecs, bytes,
                  smem_u32(&full[sidx]));
        issued = c + 1;
      }
      // After an abort, wait (bounded) for the last copy issued into each
      // stage: copies into a stage complete in issue order.
      if (*static_cast<volatile int*>(&abort_flag)) {
        for (int c = max(0, issued - kStages); c < issued; ++c)
          mbar_wait(&full[c % kStages], (c / kStages) & 1, kWaitNs, nullptr);
      }
    }
  } else {
    // Consumers.
    if (kMode == kVerify && tid == 0 && rank == 0) {
      const int tok = a.tokens[g];
      tok_ok = tok >= 0 && tok < a.V;
      if (tok_ok) {
        if (sizeof(TIn) == 2)
          x_tok = bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(row)[tok]);
        else
          x_tok = reinterpret_cast<const float*>(row)[tok];
      }
    }
    const uint32_t urow = static_cast<uint32_t>(g);
    for (int c = 0; c < nchunks; ++c) {
      const int sidx = c % kStages;
      if (!mbar_wait(&full[sidx], (c / kStages) & 1, kWaitNs, &abort_flag)) {
        if (atomicExch(&abort_flag, 1) == 0) record_error(a.err, ZARYA_DEVERR_TIMEOUT);
        break;
      }
      const int nv = min(kChunkVecs, v_hi - v_lo - c * kChunkVecs);
      const uint4* sb = stage_buf + sidx * kChunkVecs;
      // -inf in both element types, for vectors past the row
      constexpr uint32_t kNegInf = sizeof(TIn) == 2 ? 0xff80ff80u : 0xff800000u;
      uint4 v[kVecsPerThread];
#pragma unroll
      for (int k = 0; k < kVecsPerThread; ++k) {
        const int i = tid + k * kConsumers;
        v[k] = i < nv ? sb[i] : make_uint4(kNegInf, kNegInf, kNegInf, kNegInf);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[sidx]);
      const int e0 = (v_lo + c * kChunkVecs + tid) * kEpv;
      float x[kVecsPerThread][kEpv];
#pragma unroll
      for (int k = 0; k < kVecsPerThread; ++k) widen<TIn>(v[k], x[k]);
      absorb_chunk<kMode>(st, x, chunk_max<TIn>(v, x), e0, kConsumers * kEpv, a.k2);
      if (kMode == kDraftGumbel) {
        // The CTA's best score so far lets vectors that cannot win skip the
        // noise; each warp publishes its best after the stage.
        const float bound = order_float(*static_cast<volatile int*>(&best_score));
#pragma unroll
        for (int k = 0; k < kVecsPerThread; ++k)
          if (tid + k * kConsumers < nv)
            gumbel_select(st, x[k], e0 + k * kConsumers * kEpv, a, urow, bound);
        float wb = st.bz;
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) wb = fmaxf(wb, __shfl_xor_sync(0xffffffffu, wb, d));
        if (lane == 0 && wb > bound) atomicMax(&best_score, float_order(wb));
      }
    }
    // Ragged tail: V % kEpv elements, on the last rank.
    if (rank == parts - 1) {
      for (int e = nvec * kEpv + tid; e < a.V; e += kConsumers) {
        float x;
        if (sizeof(TIn) == 2)
          x = bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(row)[e]);
        else
          x = reinterpret_cast<const float*>(row)[e];
        absorb_one<kMode>(st, x, e, a, urow);
      }
    }
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) merge<kMode>(st, shfl_state<kMode>(st, d), a.k2);
    if (lane == 0) red[warp] = st;
  }
  __syncthreads();
  if (warp == 0) {
    if (lane < kConsumerWarps)
      st = red[lane];
    else
      reset(st);
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) merge<kMode>(st, shfl_state<kMode>(st, d), a.k2);
    if (lane == 0) cta_state = st;
  }
  if (parts > 1) {
    // Cluster reduction: rank 0 reads the other ranks' states; the second
    // barrier keeps their shared memory alive until it has.
    cluster_sync();
    if (rank == 0 && tid == 0) {
      const uint32_t local = smem_u32(&cta_state);
      for (int r = 1; r < parts; ++r) {
        const uint32_t ra = mapa_shared(local, static_cast<uint32_t>(r));
        RowState o;
        o.m = ld_shared_cluster_f32(ra + offsetof(RowState, m));
        o.s = ld_shared_cluster_f32(ra + offsetof(RowState, s));
        o.bz = ld_shared_cluster_f32(ra + offsetof(RowState, bz));
        o.bx = ld_shared_cluster_f32(ra + offsetof(RowState, bx));
        o.bi = __float_as_int(ld_shared_cluster_f32(ra + offsetof(RowState, bi)));
        merge<kMode>(st, o, a.k2);
      }
    }
    cluster_sync();
  }
  if (rank != 0 || tid != 0) return;

  if (kMode == kVerify) {
    if (!tok_ok) {
      record_error(a.err, ZARYA_DEVERR_TOKEN);
      a.out_prob[g] = 0.f;
    } else {
      a.out_prob[g] = ex2(lg_term(x_tok, a.k2, -st.m * a.k2)) / st.s;
    }
  } else {
    const int t = st.bi == 0x7fffffff ? 0 : st.bi;
    const float xt = kMode == kDraftGumbel ? st.bx : st.m;
    a.out_token[g] = t;
    a.out_prob[g] = ex2(lg_term(xt, a.k2, -st.m * a.k2)) / st.s;
  }
}

struct SelectArgs {
  const int32_t* n_slots;
  const int32_t* slot_len;
  const int32_t* row_offsets;
  const int32_t* draft_tokens;
  const float* draft_prob;
  float* slot_conf;
  uint8_t* slot_selected;
  int32_t* n_selected;
  int32_t* verify_row_offsets;
  int32_t* verify_src_rows;
  int32_t* verify_tokens;
  int* err;
  int B, max_slots, total_rows;
  float slot_threshold;
};

// Step 5 and the verification layout, one CTA for the whole batch, in chunks
// of kSelectThreads sequences: a warp per sequence selects its slots (lanes
// over slots), a block-wide scan places the sequences' verification rows,
// and a warp per sequence writes its row lists.
__global__ void __launch_bounds__(kSelectThreads) select_kernel(const SelectArgs a) {
  constexpr int kWarps = kSelectThreads / 32;
  __shared__ int s_count[kSelectThreads];
  __shared__ int s_pos[kSelectThreads];
  __shared__ int s_S[kSelectThreads];
  __shared__ int s_L[kSelectThreads];
  __shared__ int s_lo[kSelectThreads];
  __shared__ uint32_t s_mask[kSelectThreads];   // selected slots 0..31
  __shared__ int s_warp[kWarps];
  __shared__ int s_carry;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // The block layout was written before the row pass started (which waited
  // for it): the first chunk's is read before this kernel's wait for the
  // row pass's draws.
  int pre_S = 0, pre_L = 0, pre_lo = 0, pre_hi = 0;
  if (warp < a.B) {
    pre_S = a.n_slots[warp];
    pre_L = a.slot_len[warp];
    pre_lo = a.row_offsets[warp];
    pre_hi = a.row_offsets[warp + 1];
  }
  grid_dependency_wait();
  if (tid == 0) s_carry = 0;
  for (int b0 = 0; b0 < a.B; b0 += kSelectThreads) {
    const int nb = min(kSelectThreads, a.B - b0);
    for (int i = warp; i < nb; i += kWarps) {
      const int b = b0 + i;
      const bool pre = b0 == 0 && i == warp;
      const int S = pre ? pre_S : a.n_slots[b], L = pre ? pre_L : a.slot_len[b];
      const int lo = pre ? pre_lo : a.row_offsets[b];
      const int hi = pre ? pre_hi : a.row_offsets[b + 1];
      const bool ok = S >= 1 && L >= 1 && S <= a.max_slots && lo >= 0 && hi <= a.total_rows &&
                      static_cast<long long>(S) * L == static_cast<long long>(hi) - lo;
      float* conf = a.slot_conf + static_cast<int64_t>(b) * a.max_slots;
      uint8_t* sel = a.slot_selected + static_cast<int64_t>(b) * a.max_slots;
      int nsel = 0;
      uint32_t mask0 = 0;
      if (ok) {
        float best = -INFINITY;
        int best_s = 0x7fffffff;
        for (int s0 = 0; s0 < S; s0 += 32) {
          const int sl = s0 + lane;
          const float c = sl < S ? a.draft_prob[lo + sl * L] : -INFINITY;
          const bool take = sl < S && c > a.slot_threshold;
          const uint32_t m = __ballot_sync(0xffffffffu, take);
          nsel += __popc(m);
          if (s0 == 0) mask0 = m;
          if (sl < S) {
            conf[sl] = c;
            sel[sl] = take ? 1 : 0;
          }
          // most confident slot, first on ties
          float bc = c;
          int bs = sl < S && c > -INFINITY ? sl : 0x7fffffff;
#pragma unroll
          for (int d = 16; d >= 1; d >>= 1) {
            const float oc = __shfl_xor_sync(0xffffffffu, bc, d);
            const int os = __shfl_xor_sync(0xffffffffu, bs, d);
            if (oc > bc || (oc == bc && os < bs)) {
              bc = oc;
              bs = os;
            }
          }
          if (bc > best || (bc == best && bs < best_s)) {
            best = bc;
            best_s = bs;
          }
        }
        if (nsel == 0) {
          const int f = best_s == 0x7fffffff ? 0 : best_s;
          if (lane == 0) sel[f] = 1;
          nsel = 1;
          if (f < 32) mask0 = 1u << f;
        }
      } else if (lane == 0) {
        record_error(a.err, ZARYA_DEVERR_ROWS);
      }
      for (int s = (ok ? S : 0) + lane; s < a.max_slots; s += 32) {
        conf[s] = 0.f;
        sel[s] = 0;
      }
      if (lane == 0) {
        a.n_selected[b] = nsel;
        s_count[i] = nsel * L;
        s_S[i] = ok ? S : 0;
        s_L[i] = L;
        s_lo[i] = lo;
        s_mask[i] = mask0;
      }
    }
    __syncthreads();
    // Exclusive scan of the chunk's verification row counts.
    const int count = tid < nb ? s_count[tid] : 0;
    int incl = count;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      const int o = __shfl_up_sync(0xffffffffu, incl, d);
      if (lane >= d) incl += o;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      int w = s_warp[lane];
#pragma unroll
      for (int d = 1; d < 32; d <<= 1) {
        const int o = __shfl_up_sync(0xffffffffu, w, d);
        if (lane >= d) w += o;
      }
      s_warp[lane] = w;  // inclusive over warps
    }
    __syncthreads();
    const int carry = s_carry;
    if (tid < nb) {
      const int excl = carry + (warp > 0 ? s_warp[warp - 1] : 0) + incl - count;
      s_pos[tid] = excl;
      a.verify_row_offsets[b0 + tid] = excl;
    }
    __syncthreads();
    if (tid == 0) s_carry = carry + s_warp[kWarps - 1];
    // Row lists of the verification block: warp per sequence, slots in order.
    for (int i = warp; i < nb; i += kWarps) {
      int pos = s_pos[i];
      const int S = s_S[i], L = s_L[i], lo = s_lo[i];
      const uint8_t* sel = a.slot_selected + static_cast<int64_t>(b0 + i) * a.max_slots;
      for (int s = 0; s < S; ++s) {
        const bool taken = s < 32 ? ((s_mask[i] >> s) & 1u) != 0 : sel[s] != 0;
        if (!taken) continue;
        // pos + j < total_rows holds for non-decreasing offsets; the test
        // keeps overlapping (invalid) layouts inside the buffers.
        for (int j = lane; j < L && pos + j < a.total_rows; j += 32) {
          const int src = lo + s * L + j;
          a.verify_src_rows[pos + j] = src;
          a.verify_tokens[pos + j] = a.draft_tokens[src];
        }
        pos += L;
      }
    }
    __syncthreads();
  }
  const int total = s_carry;
  if (tid == 0) a.verify_row_offsets[a.B] = total;
  for (int k = total + tid; k < a.total_rows; k += kSelectThreads) {
    a.verify_src_rows[k] = -1;
    a.verify_tokens[k] = -1;
  }
}

struct AcceptArgs {
  const int32_t* n_slots;
  const int32_t* slot_len;
  const int32_t* row_offsets;
  const float* token_prob;
  int32_t* slot_accept;
  int32_t* accept_len;
  int* err;
  int B, max_slots, total_rows;
  float token_threshold;
};

// Step 6 acceptance: one warp per sequence.
__global__ void __launch_bounds__(kAcceptThreads) accept_kernel(const AcceptArgs a) {
  // The layout (slot counts, lengths, offsets) was written before the row
  // pass started, which waited for it: it is read before this kernel's wait
  // for the row pass's probabilities.
  const int lane = threadIdx.x & 31;
  const int b = blockIdx.x * (kAcceptThreads / 32) + (threadIdx.x >> 5);
  int S = 0, L = 0, lo = 0, hi = 0;
  if (b < a.B) {
    S = a.n_slots[b];
    L = a.slot_len[b];
    lo = a.row_offsets[b];
    hi = a.row_offsets[b + 1];
  }
  grid_dependency_wait();
  if (b >= a.B) return;
  const bool ok = S >= 0 && L >= 1 && S <= a.max_slots && lo >= 0 && hi <= a.total_rows &&
                  static_cast<long long>(S) * L == static_cast<long long>(hi) - lo;
  int32_t* sa = a.slot_accept + static_cast<int64_t>(b) * a.max_slots;
  if (!ok) {
    if (lane == 0) {
      record_error(a.err, ZARYA_DEVERR_ROWS);
      a.accept_len[b] = 0;
    }
    for (int s = lane; s < a.max_slots; s += 32) sa[s] = 0;
    return;
  }
  const float* p = a.token_prob + lo;
  const int n = S * L;
  int acc = n;
  for (int k0 = 0; k0 < n; k0 += 32) {
    const int k = k0 + lane;
    const bool fail = k < n && !(p[k] > a.token_threshold);
    const unsigned f = __ballot_sync(0xffffffffu, fail);
    if (f) {
      acc = k0 + __ffs(f) - 1;
      break;
    }
  }
  for (int s = lane; s < a.max_slots; s += 32) {
    int c = 0;
    if (s < S)
      while (c < L && p[s * L + c] > a.token_threshold) ++c;
    sa[s] = c;
  }
  if (lane == 0) a.accept_len[b] = acc;
}

template <typename TIn, int kMode>
cudaError_t launch_row_pass(const RowArgs& a, cudaStream_t stream) {
  static thread_local int configured_device = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured_device != dev) {
    e = cudaFuncSetAttribute(row_pass_kernel<TIn, kMode>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kRowSmemBytes));
    if (e != cudaSuccess) return e;
    // kRowCtasPerSm rings of stages per SM: ask for the full shared-memory carve-out.
    e = cudaFuncSetAttribute(row_pass_kernel<TIn, kMode>,
                             cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  const long long ctas = static_cast<long long>(a.total_rows) * a.parts;
  if (ctas > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  PdlLaunch l(dim3(static_cast<unsigned>(ctas)), dim3(kRowThreads), kRowSmemBytes, stream,
              static_cast<unsigned>(a.parts));
  return cudaLaunchKernelEx(&l.cfg, row_pass_kernel<TIn, kMode>, a);
}

// CTAs per row: as many as fit in one wave of resident CTAs (kRowCtasPerSm
// per SM) when the batch has few rows, at most a portable cluster (8), and at
// least two stages' worth of vectors per CTA.
int row_parts(int rows, int vocab, int elem_bytes, int sms) {
  int parts = kRowCtasPerSm * sms / max(rows, 1);
  const int nvec = static_cast<int>(static_cast<long long>(vocab) * elem_bytes / 16);
  parts = min(parts, max(1, nvec / (2 * kChunkVecs)));
  return max(1, min(parts, 8));
}

RowArgs row_args(const SampleCall& c, int* err) {
  RowArgs a{};
  a.logits = c.logits;
  a.row_stride = c.desc->row_stride;
  a.row_offsets = c.desc->row_offsets;
  a.err = err;
  a.B = c.desc->batch;
  a.V = c.desc->vocab;
  a.total_rows = c.desc->total_rows;
  const float t = c.desc->temperature;
  a.inv_t = t > 0.f ? 1.0f / t : 1.0f;
  a.k2 = t > 0.f ? kLog2e / t : kLog2e;
  a.key0 = static_cast<uint32_t>(c.desc->seed);
  a.key1 = static_cast<uint32_t>(c.desc->seed >> 32);
  a.ctr2 = static_cast<uint32_t>(c.desc->offset);
  a.ctr3 = static_cast<uint32_t>(c.desc->offset >> 32);
  a.parts = row_parts(a.total_rows, a.V, c.desc->dtype == ZARYA_BF16 ? 2 : 4, c.sms);
  return a;
}

}  // namespace

cudaError_t launch_draft_select(const SampleCall& c, const DraftOutputs& o, int* err,
                                cudaStream_t stream) {
  RowArgs a = row_args(c, err);
  a.out_token = o.draft_tokens;
  a.out_prob = o.draft_prob;
  const bool bf16 = c.desc->dtype == ZARYA_BF16;
  const bool gumbel = c.desc->temperature > 0.f;
  cudaError_t e;
  if (bf16)
    e = gumbel ? launch_row_pass<uint16_t, kDraftGumbel>(a, stream)
               : launch_row_pass<uint16_t, kDraftArgmax>(a, stream);
  else
    e = gumbel ? launch_row_pass<float, kDraftGumbel>(a, stream)
               : launch_row_pass<float, kDraftArgmax>(a, stream);
  if (e != cudaSuccess) return e;
  SelectArgs s{};
  s.n_slots = c.n_slots;
  s.slot_len = c.slot_len;
  s.row_offsets = c.desc->row_offsets;
  s.draft_tokens = o.draft_tokens;
  s.draft_prob = o.draft_prob;
  s.slot_conf = o.slot_conf;
  s.slot_selected = o.slot_selected;
  s.n_selected = o.n_selected;
  s.verify_row_offsets = o.verify_row_offsets;
  s.verify_src_rows = o.verify_src_rows;
  s.verify_tokens = o.verify_tokens;
  s.err = err;
  s.B = c.desc->batch;
  s.max_slots = c.desc->max_slots;
  s.total_rows = c.desc->total_rows;
  s.slot_threshold = c.desc->slot_threshold;
  PdlLaunch l(dim3(1), dim3(kSelectThreads), 0, stream);
  return cudaLaunchKernelEx(&l.cfg, select_kernel, s);
}

cudaError_t launch_sample_rows(const SampleCall& c, int32_t* tokens, float* prob, int* err,
                               cudaStream_t stream) {
  RowArgs a = row_args(c, err);
  a.out_token = tokens;
  a.out_prob = prob;
  const bool bf16 = c.desc->dtype == ZARYA_BF16;
  const bool gumbel = c.desc->temperature > 0.f;
  if (bf16)
    return gumbel ? launch_row_pass<uint16_t, kDraftGumbel>(a, stream)
                  : launch_row_pass<uint16_t, kDraftArgmax>(a, stream);
  return gumbel ? launch_row_pass<float, kDraftGumbel>(a, stream)
                : launch_row_pass<float, kDraftArgmax>(a, stream);
}

cudaError_t launch_verify_accept(const SampleCall& c, const int32_t* tokens, float* token_prob,
                                 int32_t* slot_accept, int32_t* accept_len, int* err,
                                 cudaStream_t stream) {
  RowArgs a = row_args(c, err);
  a.tokens = tokens;
  a.out_prob = token_prob;
  cudaError_t e = c.desc->dtype == ZARYA_BF16 ? launch_row_pass<uint16_t, kVerify>(a, stream)
                                              : launch_row_pass<float, kVerify>(a, stream);
  if (e != cudaSuccess) return e;
  AcceptArgs s{};
  s.n_slots = c.n_slots;
  s.slot_len = c.slot_len;
  s.row_offsets = c.desc->row_offsets;
  s.token_prob = token_prob;
  s.slot_accept = slot_accept;
  s.accept_len = accept_len;
  s.err = err;
  s.B = c.desc->batch;
  s.max_slots = c.desc->max_slots;
  s.total_rows = c.desc->total_rows;
  s.token_threshold = c.desc->token_threshold;
  const int per = kAcceptThreads / 32;
  PdlLaunch l(dim3(static_cast<unsigned>((c.desc->batch + per - 1) / per)), dim3(kAcceptThreads),
              0, stream);
  return cudaLaunchKernelEx(&l.cfg, accept_kernel, s);
}

}  // namespace zarya
