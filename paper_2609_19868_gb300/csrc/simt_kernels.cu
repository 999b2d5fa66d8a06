// CUDA-core kernels of the library:
//   * slot attention in true fp32 (the fp32 storage type; tensor-core tf32
//     would not meet fp32 accuracy), one warp per (sequence, query head, row);
//   * KV append of accepted tokens (Sec. 5.2 step 7): 16-byte vector copies of
//     whole token rows (Hkv * D contiguous elements) into the cache, through
//     the page table when paged, followed by the length advance;
//   * the per-device error word.
#include <cuda_runtime.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace zarya {

// One error word per device that loads the library (zero = no error).
__device__ int g_error_word = 0;

int* device_error_word(cudaError_t* status) {
  constexpr int kMaxDevices = 64;
  static int* cache[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
    if (status) *status = (e != cudaSuccess) ? e : cudaErrorInvalidDevice;
    return nullptr;
  }
  int* ptr = __atomic_load_n(&cache[dev], __ATOMIC_ACQUIRE);
  if (ptr == nullptr) {
    e = cudaGetSymbolAddress(reinterpret_cast<void**>(&ptr), g_error_word);
    if (e != cudaSuccess) {
      if (status) *status = e;
      return nullptr;
    }
    __atomic_store_n(&cache[dev], ptr, __ATOMIC_RELEASE);
  }
  if (status) *status = cudaSuccess;
  return ptr;
}

namespace {

// Validates sequence b of an attention call; returns its error code or 0.
__device__ __forceinline__ int check_sequence(const SimtParams& p, int b, int* P_out, int* R_out,
                                              int* mode_out, int* row0_out) {
  const int P = p.cache_lens[b];
  // R_b = S_b * L_b, clamped so that an absurd product reads as invalid below
  const long long R64 = static_cast<long long>(p.n_slots[b]) * p.slot_len[b];
  const int R = R64 > p.max_rows ? p.max_rows + 1 : static_cast<int>(R64);
  const int mode = p.mask_mode[b];
  const int row0 = p.q_row_offsets[b];
  const int row_end = p.q_row_offsets[b + 1];
  *P_out = P;
  *R_out = R;
  *mode_out = mode;
  *row0_out = row0;
  if (mode != ZARYA_MASK_BIDIR_BLOCK && mode != ZARYA_MASK_SLOT_CAUSAL &&
      mode != ZARYA_MASK_SLOT_INDEPENDENT)
    return ZARYA_DEVERR_MASK_MODE;
  if (p.n_slots[b] < 1 || p.slot_len[b] < 1 || R > p.max_rows || row_end - row0 != R ||
      row0 < 0 || row_end > p.total_rows)
    return ZARYA_DEVERR_ROWS;
  if (P < 0 || static_cast<long long>(P) + R > p.capacity) return ZARYA_DEVERR_CAPACITY;
  return 0;
}

// Token row index (in units of Hkv * D elements) of logical token c of
// sequence b, or -1 when the page id is out of range.
__device__ __forceinline__ long long token_row(const int32_t* page_table, int page_size,
                                               int max_pages, int n_pages, int capacity, int b,
                                               int c) {
  if (page_size == 0) return static_cast<long long>(b) * capacity + c;
  const int page = page_table[static_cast<long long>(b) * max_pages + c / page_size];
  if (page < 0 || page >= n_pages) return -1;
  return static_cast<long long>(page) * page_size + c % page_size;
}

constexpr int kF32Warps = 8;   // warps per CTA of the fp32 attention kernel

// One CTA per (sequence, head, block row). The row's visible keys (the
// earlier slots' hidden block rows [P, hide_hi) skipped) go in chunks of 32 to
// the CTA's warps in turn; within a chunk lane k scores key k with a whole
// dot product, the warp takes the chunk's maximum and sum and broadcasts the
// weights to accumulate O (lane l holds columns l, l + 32, ...), an online
// softmax over the warp's chunks. The warps' partial (m, l, O) then merge in
// shared memory: O = sum_w e^(m_w - M) O_w / sum_w e^(m_w - M) l_w.
template <int kPerLane>
__global__ void __launch_bounds__(kF32Warps * 32)
slot_attn_f32_kernel(const SimtParams p) {
  grid_dependency_wait();
  grid_launch_dependents();
  constexpr int D = kPerLane * 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const long long per_b = static_cast<long long>(p.Hq) * p.max_rows;
  const int b = static_cast<int>(blockIdx.x / per_b);
  if (b >= p.B) return;
  const int rem = static_cast<int>(blockIdx.x - b * per_b);
  const int h = rem / p.max_rows;
  const int r = rem - h * p.max_rows;
  int P, R, mode, row0;
  const int code = check_sequence(p, b, &P, &R, &mode, &row0);
  if (code != 0) {
    if (h == 0 && r == 0 && threadIdx.x == 0) record_error(p.err, code);
    return;
  }
  if (r >= R) return;   // uniform over the CTA
  const int g = p.Hq / p.Hkv;
  const int j = h / g;
  const int n_vis = (mode == ZARYA_MASK_BIDIR_BLOCK) ? P + R : P + r + 1;
  // slot-independent: the earlier slots' block rows [P, P + s L) are hidden
  const int hide_hi = (mode == ZARYA_MASK_SLOT_INDEPENDENT) ? P + (r / p.slot_len[b]) * p.slot_len[b] : P;
  const float* q = reinterpret_cast<const float*>(p.q) +
                   (static_cast<long long>(row0 + r) * p.Hq + h) * D;
  const float* kc = reinterpret_cast<const float*>(p.k_cache);
  const float* vc = reinterpret_cast<const float*>(p.v_cache);
  __shared__ float4 qs[D / 4];                 // the query row (every lane reads all of it)
  __shared__ float s_o[kF32Warps][D];          // the warps' partial outputs
  __shared__ float s_m[kF32Warps], s_l[kF32Warps];
  __shared__ int s_bad;
  if (threadIdx.x == 0) s_bad = 0;
  for (int i = threadIdx.x; i < D; i += kF32Warps * 32) reinterpret_cast<float*>(qs)[i] = q[i];
  __syncthreads();
  const int nv = P + (n_vis - hide_hi);
  float o[kPerLane];
#pragma unroll
  for (int x = 0; x < kPerLane; ++x) o[x] = 0.f;
  float m = -INFINITY, l = 0.f;
  for (int base = warp * 32; base < nv; base += kF32Warps * 32) {
    const int i = base + lane;
    float s = -INFINITY;
    long long row = 0;   // first element of this lane's key row (K and V)
    bool bad = false;
    if (i < nv) {
      const int c = i < P ? i : i - P + hide_hi;
      const long long tr =
          token_row(p.page_table, p.page_size, p.max_pages, p.n_pages, p.capacity, b, c);
      if (tr < 0) {
        bad = true;
      } else {
        row = (tr * p.Hkv + j) * D;
        const float4* k4 = reinterpret_cast<const float4*>(kc + row);
        float dot0 = 0.f, dot1 = 0.f;
#pragma unroll 8
        for (int d = 0; d < D / 4; ++d) {
          const float4 kv = k4[d];
          const float4 qv = qs[d];
          dot0 = fmaf(qv.x, kv.x, dot0);
          dot1 = fmaf(qv.y, kv.y, dot1);
          dot0 = fmaf(qv.z, kv.z, dot0);
          dot1 = fmaf(qv.w, kv.w, dot1);
        }
        s = (dot0 + dot1) * p.scale;
      }
    }
    if (__any_sync(0xffffffffu, bad)) {
      if (lane == 0) s_bad = 1;
      break;
    }
    float cm = s;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, off));
    const float m_new = fmaxf(m, cm);
    const float corr = (m == -INFINITY) ? 0.f : expf(m - m_new);
    const float w = (i < nv) ? expf(s - m_new) : 0.f;
    float ws = w;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ws += __shfl_xor_sync(0xffffffffu, ws, off);
    l = l * corr + ws;
#pragma unroll
    for (int x = 0; x < kPerLane; ++x) o[x] *= corr;
    const int n = min(32, nv - base);
#pragma unroll 16
    for (int k = 0; k < 32; ++k) {
      const float wk = __shfl_sync(0xffffffffu, w, k);
      const long long rk = __shfl_sync(0xffffffffu, row, k);
      if (k < n) {
#pragma unroll
        for (int x = 0; x < kPerLane; ++x) o[x] = fmaf(wk, vc[rk + lane + 32 * x], o[x]);
      }
    }
    m = m_new;
  }
  if (lane == 0) {
    s_m[warp] = m;
    s_l[warp] = l;
  }
#pragma unroll
  for (int x = 0; x < kPerLane; ++x) s_o[warp][lane + 32 * x] = o[x];
  __syncthreads();
  if (s_bad) {
    if (threadIdx.x == 0) record_error(p.err, ZARYA_DEVERR_PAGE_ID);
    return;
  }
  float M = -INFINITY;
#pragma unroll
  for (int w = 0; w < kF32Warps; ++w) M = fmaxf(M, s_m[w]);
  float L = 0.f;
  float wt[kF32Warps];
#pragma unroll
  for (int w = 0; w < kF32Warps; ++w) {
    wt[w] = (s_m[w] == -INFINITY) ? 0.f : expf(s_m[w] - M);
    L = fmaf(wt[w], s_l[w], L);
  }
  float* out = reinterpret_cast<float*>(p.out) + (static_cast<long long>(row0 + r) * p.Hq + h) * D;
  for (int t = threadIdx.x; t < D; t += kF32Warps * 32) {
    float acc = 0.f;
#pragma unroll
    for (int w = 0; w < kF32Warps; ++w) acc = fmaf(wt[w], s_o[w][t], acc);
    out[t] = acc / L;
  }
}

// At most this many CTAs share one sequence's rows, so that a commit can
// advance cache_lens[b] inside one thread-block cluster.
constexpr int kAppendMaxCtasPerSeq = 8;
constexpr int kAppendThreads = 256;
constexpr int kCommitThreads = 128;
constexpr int kAppendUnroll = 4;   // 16-byte vectors of K and of V in flight per thread

// Copies rows i < accept_len[b] of the block (rows [x * rows_per_block, ...)
// for CTA x, sequence blockIdx.y) to cache positions P_b + i. With `commit`
// the CTAs of a sequence form one cluster: after every CTA has read P_b and
// copied its rows, CTA 0 writes new_lens[b] = P_b + accept_len[b].
template <bool kCommit>
__global__ void __launch_bounds__(kAppendThreads)
kv_append_copy_kernel(const AppendParams p) {
  grid_dependency_wait();
  grid_launch_dependents();
  const int b = blockIdx.y;
  const int P = p.cache_lens[b];
  const int row0 = p.q_row_offsets[b];
  const int R = p.q_row_offsets[b + 1] - row0;
  const int a = p.accept_len != nullptr ? p.accept_len[b] : R;   // nullptr: the whole block
  int code = 0;
  if (R < 0 || R > p.max_rows || row0 < 0 || row0 + R > p.total_rows) code = ZARYA_DEVERR_ROWS;
  else if (a < 0 || a > R) code = ZARYA_DEVERR_ACCEPT;
  else if (P < 0 || static_cast<long long>(P) + a > p.capacity) code = ZARYA_DEVERR_CAPACITY;
  if (code != 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(p.err, code);
  } else {
    const int i0 = blockIdx.x * p.rows_per_block;
    const int n_rows = max(0, min(p.rows_per_block, a - i0));
    const int vec_per_row = p.row_bytes >> 4;
    const uint4* kn = reinterpret_cast<const uint4*>(p.k_new);
    const uint4* vn = reinterpret_cast<const uint4*>(p.v_new);
    uint4* kc = reinterpret_cast<uint4*>(p.k_cache);
    uint4* vc = reinterpret_cast<uint4*>(p.v_cache);
    const int total = n_rows * vec_per_row;
    for (int base = 0; base < total; base += kAppendUnroll * kAppendThreads) {
      uint4 kv[kAppendUnroll], vv[kAppendUnroll];
      long long dst[kAppendUnroll];
      // all loads first, then all stores: kAppendUnroll round trips overlap
#pragma unroll
      for (int u = 0; u < kAppendUnroll; ++u) {
        const int idx = base + u * kAppendThreads + threadIdx.x;
        dst[u] = -1;
        if (idx < total) {
          const int ri = idx / vec_per_row;
          const int v = idx - ri * vec_per_row;
          const int i = i0 + ri;
          const int t = P + i;
          long long tr = -1;
          if (p.page_size == 0) {
            tr = static_cast<long long>(b) * p.capacity + t;
          } else {
            const int page = p.page_table[static_cast<long long>(b) * p.max_pages + t / p.page_size];
            if (page < 0 || page >= p.n_pages) record_error(p.err, ZARYA_DEVERR_PAGE_ID);
            else tr = static_cast<long long>(page) * p.page_size + t % p.page_size;
          }
          if (tr >= 0) {
            const long long src = static_cast<long long>(row0 + i) * vec_per_row + v;
            kv[u] = __ldg(kn + src);
            vv[u] = __ldg(vn + src);
            dst[u] = tr * vec_per_row + v;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kAppendUnroll; ++u) {
        if (dst[u] >= 0) {
          kc[dst[u]] = kv[u];
          vc[dst[u]] = vv[u];
        }
      }
    }
  }
  if (kCommit) {
    // Every CTA of this sequence has read cache_lens[b] before it changes
    // (new_lens may alias cache_lens).
    cluster_arrive();
    cluster_wait();
    if (code == 0 && blockIdx.x == 0 && threadIdx.x == 0) p.new_lens[b] = P + a;
  }
}

// Commit of a block whose rows the verification pass already staged at
// positions P_b.. (Sec. 5.2 step 7 with nothing left to copy): one thread per
// sequence checks accept_len[b] and writes new_lens[b] = P_b + accept_len[b].
// It waits for the kernel before it (accept_len comes from the acceptance
// step, and new_lens may be the cache_lens that kernel reads).
__global__ void __launch_bounds__(kCommitThreads) commit_lens_kernel(const AppendParams p) {
  grid_dependency_wait();
  grid_launch_dependents();
  const int b = blockIdx.x * kCommitThreads + threadIdx.x;
  if (b >= p.B) return;
  const int P = p.cache_lens[b];
  const int row0 = p.q_row_offsets[b];
  const int R = p.q_row_offsets[b + 1] - row0;
  const int a = p.accept_len[b];
  int code = 0;
  if (R < 0 || R > p.max_rows || row0 < 0 || row0 + R > p.total_rows) code = ZARYA_DEVERR_ROWS;
  else if (a < 0 || a > R) code = ZARYA_DEVERR_ACCEPT;
  else if (P < 0 || static_cast<long long>(P) + a > p.capacity) code = ZARYA_DEVERR_CAPACITY;
  if (code != 0) record_error(p.err, code);
  else p.new_lens[b] = P + a;
}

}  // namespace

cudaError_t launch_commit_lens(const AppendParams& p, cudaStream_t stream) {
  PdlLaunch l(dim3(static_cast<unsigned>((p.B + kCommitThreads - 1) / kCommitThreads)),
              dim3(kCommitThreads), 0, stream);
  return cudaLaunchKernelEx(&l.cfg, commit_lens_kernel, p);
}

cudaError_t launch_slot_attn_f32(const SimtParams& p, cudaStream_t stream) {
  const long long grid = static_cast<long long>(p.B) * p.Hq * p.max_rows;   // one CTA per row
  if (grid > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
  PdlLaunch l(dim3(static_cast<unsigned>(grid)), dim3(kF32Warps * 32), 0, stream);
  switch (p.D / 32) {
    case 1: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<1>, p);
    case 2: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<2>, p);
    case 3: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<3>, p);
    case 4: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<4>, p);
    case 5: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<5>, p);
    case 6: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<6>, p);
    case 7: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<7>, p);
    case 8: return cudaLaunchKernelEx(&l.cfg, slot_attn_f32_kernel<8>, p);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_kv_append(const AppendParams& p_in, bool commit, cudaStream_t stream) {
  AppendParams p = p_in;
  const int rows = p.max_rows > 0 ? p.max_rows : 1;
  p.rows_per_block = max(8, (rows + kAppendMaxCtasPerSeq - 1) / kAppendMaxCtasPerSeq);
  const int ctas = (rows + p.rows_per_block - 1) / p.rows_per_block;   // <= 8
  if (commit) {
    PdlLaunch l(dim3(ctas, p.B), dim3(kAppendThreads), 0, stream, static_cast<unsigned>(ctas));
    return cudaLaunchKernelEx(&l.cfg, kv_append_copy_kernel<true>, p);
  }
  PdlLaunch l(dim3(ctas, p.B), dim3(kAppendThreads), 0, stream);
  return cudaLaunchKernelEx(&l.cfg, kv_append_copy_kernel<false>, p);
}

}  // namespace zarya
