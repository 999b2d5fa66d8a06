// Slot attention on the sm_103a tensor cores (bf16 in, fp32 accumulate).
//
// Computes Zarya's Mode B attention step (Sec. 5.2, step 3 draft pass with a
// block-bidirectional mask and step 6 verification pass with a causal mask
// over the reordered sequence): each block row of sequence b attends over the
// committed prefix in the KV cache plus the block's own keys staged after it.
//
// One CTA owns one work tile (sequence b, KV head j, M-tile, KV split):
//   * M = 128 packed rows: the GQA group of g = Hq/Hkv query heads times
//     128/g block rows (packed row m -> block row r0 + m/g, head j*g + m%g),
//     loaded by one 3-D TMA box per 64-column half of Q;
//   * keys stream through shared memory in tiles of 128 (TMA, 128-byte
//     swizzle; paged caches use one box per page);
//   * S = Q K^T goes to TMEM (double buffered, 2 x 128 columns) via
//     tcgen05.mma issued by one thread; softmax warps read S with
//     tcgen05.ld, apply the mask from indices, run the online softmax (exp2
//     on the MUFU), write P (bf16) to shared memory; O += P V accumulates in
//     TMEM (128 columns);
//   * when the key range is split across CTAs, each writes a normalised
//     partial (O_i, log2-sum-exp_i) to the workspace and the last CTA to
//     arrive merges them: O = sum_i 2^(lse_i - lse_max) O_i / sum_i 2^(...).
//
// Warp roles (256 threads): warp 0 TMA producer, warp 1 MMA issuer, warp 2
// TMEM allocator, warp 3 idle, warps 4-7 softmax + epilogue (warp w reads
// TMEM lanes 32*(w%4) .. +31, i.e. packed rows of that range).
//
// Every mbarrier wait is bounded (about 2 s of global time); a wait that
// gives up records ZARYA_DEVERR_TIMEOUT, raises a CTA-wide abort flag and the
// CTA unwinds (draining its own copies and MMAs, freeing TMEM).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace zarya {
namespace {

constexpr int kThreads = 256;
constexpr int kStagesK = 3;
constexpr int kStagesV = 2;
constexpr uint32_t kHalfBytes = kBlockN * 64 * 2;   // 128 rows x 128 B
constexpr uint32_t kTileBytes = 2 * kHalfBytes;     // 32 KB (128 x 128 bf16)
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kTileBytes;
constexpr uint32_t kOffV = kOffK + kStagesK * kTileBytes;
constexpr uint32_t kOffP = kOffV + kStagesV * kTileBytes;
constexpr uint32_t kOffBar = kOffP + kTileBytes;
constexpr uint32_t kTmemCols = 512;                 // S0 [0,128) S1 [128,256) O [256,384)
constexpr uint32_t kTmemO = 256;
constexpr uint64_t kWaitNs = 2000000000ull;         // 2 s
constexpr uint64_t kDrainNs = 100000000ull;         // 100 ms

struct Bars {
  uint64_t q_full;
  uint64_t k_full[kStagesK];
  uint64_t k_empty[kStagesK];
  uint64_t v_full[kStagesV];
  uint64_t v_empty[kStagesV];
  uint64_t s_full[2];
  uint64_t s_free[2];
  uint64_t p_full;
  uint64_t o_done;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  int last;
};

constexpr uint32_t kSmemBytes = kOffBar + ((sizeof(Bars) + 127) / 128) * 128 + 1024;
static_assert(kSmemBytes <= 232448, "shared memory budget");

constexpr uint32_t kIdescQK = idesc_bf16_f32(128, 128, false, false);
constexpr uint32_t kIdescPV = idesc_bf16_f32(128, 128, false, true);

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void named_bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

__device__ __forceinline__ void set_abort(Bars* bars, int* err, int code) {
  record_error(err, code);
  *reinterpret_cast<volatile int*>(&bars->abort) = 1;
}

__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, Bars* bars, int* err) {
  if (mbar_wait(bar, parity, kWaitNs, &bars->abort)) return true;
  set_abort(bars, err, ZARYA_DEVERR_TIMEOUT);
  return false;
}

// Offset (bytes) of the k-th 16-element K slice inside a 128-row, 2-half,
// K-major SW128 tile.
__device__ __forceinline__ uint32_t kmajor_k_offset(int kk) {
  return (kk >> 2) * kHalfBytes + (kk & 3) * 32;
}

__global__ void __launch_bounds__(kThreads, 1)
slot_attn_tc_kernel(const __grid_constant__ CUtensorMap map_q,
                    const __grid_constant__ CUtensorMap map_k,
                    const __grid_constant__ CUtensorMap map_v, const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + kOffBar);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int mt = blockIdx.x;
  const int split = blockIdx.y;
  const int bh = blockIdx.z;
  const int b = bh / p.Hkv;
  const int kvh = bh - b * p.Hkv;

  // ---- per-sequence geometry (uniform over the CTA) ----
  const int P = p.cache_lens[b];
  const int R = p.n_slots[b] * p.slot_len[b];
  const int mode = p.mask_mode[b];
  const int row0 = p.q_row_offsets[b];
  const int row_end = p.q_row_offsets[b + 1];
  int code = 0;
  if (mode != ZARYA_MASK_BIDIR_BLOCK && mode != ZARYA_MASK_SLOT_CAUSAL) code = ZARYA_DEVERR_MASK_MODE;
  else if (R <= 0 || R > p.max_rows || row_end - row0 != R || row0 < 0 || row_end > p.total_rows)
    code = ZARYA_DEVERR_ROWS;
  else if (P < 0 || static_cast<long long>(P) + R > p.capacity) code = ZARYA_DEVERR_CAPACITY;
  if (code != 0) {
    if (mt == 0 && split == 0 && threadIdx.x == 0) record_error(p.err, code);
    return;
  }
  const int rows_per_tile = kBlockM / p.g;
  const int r0 = mt * rows_per_tile;
  if (r0 >= R) return;
  const int r_hi = min(r0 + rows_per_tile, R) - 1;
  const int kv_end = (mode == ZARYA_MASK_SLOT_CAUSAL) ? P + r_hi + 1 : P + R;
  const int n_tiles = (kv_end + kBlockN - 1) / kBlockN;
  const int per_split = (n_tiles + p.splits - 1) / p.splits;
  const int active = (n_tiles + per_split - 1) / per_split;
  if (split >= active) return;
  const int t_begin = split * per_split;
  const int nt = min(n_tiles, t_begin + per_split) - t_begin;
  const bool paged = p.page_size > 0;

  // ---- set-up ----
  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    for (int s = 0; s < kStagesK; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], 1);
    }
    for (int s = 0; s < kStagesV; ++s) {
      mbar_init(&bars->v_full[s], 1);
      mbar_init(&bars->v_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars->s_full[s], 1);
      mbar_init(&bars->s_free[s], 4);
    }
    mbar_init(&bars->p_full, 4);
    mbar_init(&bars->o_done, 1);
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    bars->last = 0;
    fence_mbar_init();
  }
  if (warp == 2) {
    tmem_alloc(&bars->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_q);
    tma_prefetch_map(&map_k);
    tma_prefetch_map(&map_v);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;

  if (warp == 0) {
    // ======================= TMA producer =======================
    int issued_k = 0, issued_v = 0;
    bool ok = true;
    if (lane == 0) {
      mbar_arrive_expect_tx(&bars->q_full, kTileBytes);
      const uint32_t dq = smem_u32(smem + kOffQ);
      tma_load_3d(dq, &map_q, &bars->q_full, 0, kvh * p.g, row0 + r0);
      tma_load_3d(dq + kHalfBytes, &map_q, &bars->q_full, 64, kvh * p.g, row0 + r0);
    }
    const int ppt = paged ? kBlockN / p.page_size : 0;   // pages per tile
    const uint32_t page_bytes = paged ? static_cast<uint32_t>(p.page_size) * 256u : 0u;
    for (int i = 0; i < nt && ok; ++i) {
      const int t = t_begin + i;
      // page ids of this tile: lane l < ppt owns page l
      int page = -1;
      uint32_t bytes = kTileBytes;
      if (paged) {
        const int lp = t * ppt + lane;
        const bool want = lane < ppt && lp * p.page_size < kv_end;
        bool bad = false;
        if (want) {
          page = p.page_table[static_cast<long long>(b) * p.max_pages + lp];
          bad = page < 0 || page >= p.n_pages;
        }
        if (__any_sync(0xffffffffu, bad)) {
          if (lane == 0) set_abort(bars, p.err, ZARYA_DEVERR_PAGE_ID);
          ok = false;
          break;
        }
        bytes = page_bytes * __popc(__ballot_sync(0xffffffffu, want));
      }
      // K tile
      {
        const int s = i % kStagesK;
        const uint32_t ph = (i / kStagesK) & 1;
        bool w = true;
        if (lane == 0) {
          w = wait_bar(&bars->k_empty[s], ph ^ 1, bars, p.err);
          if (w) mbar_arrive_expect_tx(&bars->k_full[s], bytes);
        }
        if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
        issued_k = i + 1;
        const uint32_t dst = smem_u32(smem + kOffK + s * kTileBytes);
        if (!paged) {
          if (lane == 0) {
            tma_load_4d(dst, &map_k, &bars->k_full[s], 0, kvh, t * kBlockN, b);
            tma_load_4d(dst + kHalfBytes, &map_k, &bars->k_full[s], 64, kvh, t * kBlockN, b);
          }
        } else if (page >= 0) {
          const uint32_t o = lane * p.page_size * 128;
          tma_load_4d(dst + o, &map_k, &bars->k_full[s], 0, kvh, 0, page);
          tma_load_4d(dst + kHalfBytes + o, &map_k, &bars->k_full[s], 64, kvh, 0, page);
        }
      }
      // V tile
      {
        const int s = i % kStagesV;
        const uint32_t ph = (i / kStagesV) & 1;
        bool w = true;
        if (lane == 0) {
          w = wait_bar(&bars->v_empty[s], ph ^ 1, bars, p.err);
          if (w) mbar_arrive_expect_tx(&bars->v_full[s], bytes);
        }
        if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
        issued_v = i + 1;
        const uint32_t dst = smem_u32(smem + kOffV + s * kTileBytes);
        if (!paged) {
          if (lane == 0) {
            tma_load_4d(dst, &map_v, &bars->v_full[s], 0, kvh, t * kBlockN, b);
            tma_load_4d(dst + kHalfBytes, &map_v, &bars->v_full[s], 64, kvh, t * kBlockN, b);
          }
        } else if (page >= 0) {
          const uint32_t o = lane * p.page_size * 128;
          tma_load_4d(dst + o, &map_v, &bars->v_full[s], 0, kvh, 0, page);
          tma_load_4d(dst + kHalfBytes + o, &map_v, &bars->v_full[s], 64, kvh, 0, page);
        }
      }
    }
    if (!ok && lane == 0) {
      // Let this CTA's own copies land before the CTA (and its smem) goes away.
      for (int i = max(0, issued_k - kStagesK); i < issued_k; ++i)
        mbar_wait(&bars->k_full[i % kStagesK], (i / kStagesK) & 1, kDrainNs, nullptr);
      for (int i = max(0, issued_v - kStagesV); i < issued_v; ++i)
        mbar_wait(&bars->v_full[i % kStagesV], (i / kStagesV) & 1, kDrainNs, nullptr);
      mbar_wait(&bars->q_full, 0, kDrainNs, nullptr);
    }
  } else if (warp == 1) {
    // ======================= MMA issuer (one thread) =======================
    if (lane == 0) {
      bool ok = wait_bar(&bars->q_full, 0, bars, p.err);
      bool any_mma = false;
      tc_fence_after();
      const uint32_t q_addr = smem_u32(smem + kOffQ);
      const uint32_t p_addr = smem_u32(smem + kOffP);
      auto issue_pv = [&](int j) -> bool {
        const int sv = j % kStagesV;
        if (!wait_bar(&bars->p_full, j & 1, bars, p.err)) return false;
        if (!wait_bar(&bars->v_full[sv], (j / kStagesV) & 1, bars, p.err)) return false;
        tc_fence_after();
        const uint32_t v_addr = smem_u32(smem + kOffV + sv * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t ad = sdesc_sw128(p_addr + kmajor_k_offset(kk), 16, 1024);
          const uint64_t bd = sdesc_sw128(v_addr + kk * 2048, kHalfBytes, 1024);
          tc_mma_ss(tmem + kTmemO, ad, bd, kIdescPV, (j > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(&bars->o_done);
        tc_commit(&bars->v_empty[sv]);
        return true;
      };
      for (int i = 0; i < nt && ok; ++i) {
        const int s = i % kStagesK;
        const int sb = i & 1;
        if (!wait_bar(&bars->k_full[s], (i / kStagesK) & 1, bars, p.err)) { ok = false; break; }
        if (!wait_bar(&bars->s_free[sb], ((i >> 1) & 1) ^ 1, bars, p.err)) { ok = false; break; }
        tc_fence_after();
        const uint32_t k_addr = smem_u32(smem + kOffK + s * kTileBytes);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t ad = sdesc_sw128(q_addr + kmajor_k_offset(kk), 16, 1024);
          const uint64_t bd = sdesc_sw128(k_addr + kmajor_k_offset(kk), 16, 1024);
          tc_mma_ss(tmem + sb * 128, ad, bd, kIdescQK, kk > 0 ? 1u : 0u);
        }
        any_mma = true;
        tc_commit(&bars->s_full[sb]);
        tc_commit(&bars->k_empty[s]);
        if (i > 0 && !issue_pv(i - 1)) { ok = false; break; }
      }
      if (ok && nt > 0) ok = issue_pv(nt - 1);
      if (!ok && any_mma) {
        tc_commit(&bars->drain);
        mbar_wait(&bars->drain, 0, kDrainNs, nullptr);
      }
    }
  } else if (warp >= 4) {
    // ======================= softmax + epilogue =======================
    const int wq = warp & 3;
    const int m = wq * 32 + lane;                   // packed row = TMEM lane
    const int r = r0 + m / p.g;
    const int h = kvh * p.g + (m - (m / p.g) * p.g);
    const bool row_ok = r <= r_hi;
    const int limit = !row_ok ? kv_end : (mode == ZARYA_MASK_SLOT_CAUSAL ? P + r + 1 : P + R);
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(wq * 32) << 16);
    const float sl2 = p.scale_log2;
    float m_run = -INFINITY;  // running max, in scaled log2 units
    float l_run = 0.f;
    bool ok = true;
    uint8_t* sp = smem + kOffP;

    for (int i = 0; i < nt; ++i) {
      const int c0 = (t_begin + i) * kBlockN;
      const int sb = i & 1;
      if (ok) ok = wait_bar(&bars->s_full[sb], (i >> 1) & 1, bars, p.err);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      float s[128];
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) {
        float v[32];
        tmem_ld_32x32b_x32(t_lane + sb * 128 + ch * 32, v);
#pragma unroll
        for (int x = 0; x < 32; ++x) s[ch * 32 + x] = v[x];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->s_free[sb]);

      if (c0 + kBlockN > limit) {
#pragma unroll
        for (int x = 0; x < 128; ++x)
          if (c0 + x >= limit) s[x] = -INFINITY;
      }
      float mx = -INFINITY;
#pragma unroll
      for (int x = 0; x < 128; ++x) mx = fmaxf(mx, s[x]);
      const float m_new = fmaxf(m_run, mx * sl2);
      const bool need = m_new > m_run + 8.0f;
      const bool warp_need = __any_sync(0xffffffffu, need);
      float alpha = 1.f;
      if (warp_need) {
        alpha = (m_run == -INFINITY) ? 0.f : fast_exp2(m_run - m_new);
        m_run = m_new;
        l_run *= alpha;
      }
      const float m_use = (m_run == -INFINITY) ? 0.f : m_run;
      uint32_t pk[64];
      float rs = 0.f;
#pragma unroll
      for (int x = 0; x < 128; x += 2) {
        const float p0 = fast_exp2(fmaf(s[x], sl2, -m_use));
        const float p1 = fast_exp2(fmaf(s[x + 1], sl2, -m_use));
        rs += p0 + p1;
        pk[x >> 1] = pack_bf16(p0, p1);
      }
      l_run += rs;

      // Keys at or past kv_end in the last tile: their V rows (stale smem,
      // unloaded pages or another sequence's cache) must be exact zeros, or a
      // NaN there would poison P*V even with P = 0.
      if (c0 + kBlockN > kv_end) {
        const int sv = i % kStagesV;
        if (ok) ok = wait_bar(&bars->v_full[sv], (i / kStagesV) & 1, bars, p.err);
        if (ok && c0 + m >= kv_end) {
          uint8_t* vrow = smem + kOffV + sv * kTileBytes + (m >> 3) * 1024 + (m & 7) * 128;
          const uint4 z = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
          for (int x = 0; x < 8; ++x) {
            reinterpret_cast<uint4*>(vrow)[x] = z;
            reinterpret_cast<uint4*>(vrow + kHalfBytes)[x] = z;
          }
        }
      }
      // P of the previous tile must have been consumed (and O be final for
      // the rescale) before P is overwritten.
      if (i > 0) {
        if (ok) ok = wait_bar(&bars->o_done, (i - 1) & 1, bars, p.err);
        tc_fence_after();
      }
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      if (warp_need && i > 0) {
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          float v[32];
          const uint32_t a = t_lane + kTmemO + ch * 32;
          tmem_ld_32x32b_x32(a, v);
#pragma unroll
          for (int x = 0; x < 32; ++x) v[x] *= alpha;
          tmem_st_32x32b_x32(a, v);
        }
      }
      uint8_t* prow = sp + (m >> 3) * 1024 + (m & 7) * 128;
#pragma unroll
      for (int c16 = 0; c16 < 16; ++c16) {
        const uint32_t off = (c16 >> 3) * kHalfBytes + ((((c16 & 7) ^ (m & 7))) << 4);
        *reinterpret_cast<uint4*>(prow + off) =
            make_uint4(pk[c16 * 4 + 0], pk[c16 * 4 + 1], pk[c16 * 4 + 2], pk[c16 * 4 + 3]);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->p_full);
    }

    // ---- epilogue ----
    if (ok) ok = wait_bar(&bars->o_done, (nt - 1) & 1, bars, p.err);
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();
    const long long unit = static_cast<long long>(bh) * p.m_tiles + mt;
    if (active == 1) {
      const float inv = (l_run > 0.f) ? 1.f / l_run : 0.f;
      __nv_bfloat16* dst = reinterpret_cast<__nv_bfloat16*>(p.out) +
                           (static_cast<long long>(row0 + r) * p.Hq + h) * kHeadDim;
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) {
        float v[32];
        if (ok) tmem_ld_32x32b_x32(t_lane + kTmemO + ch * 32, v);
        if (ok && row_ok) {
          uint4* d4 = reinterpret_cast<uint4*>(dst + ch * 32);
#pragma unroll
          for (int x = 0; x < 4; ++x)
            d4[x] = make_uint4(pack_bf16(v[8 * x + 0] * inv, v[8 * x + 1] * inv),
                               pack_bf16(v[8 * x + 2] * inv, v[8 * x + 3] * inv),
                               pack_bf16(v[8 * x + 4] * inv, v[8 * x + 5] * inv),
                               pack_bf16(v[8 * x + 6] * inv, v[8 * x + 7] * inv));
        }
      }
    } else {
      const float inv = (l_run > 0.f) ? 1.f / l_run : 0.f;
      const long long slot = (unit * p.splits + split) * kBlockM + m;
      float* po = p.ws_o + slot * kHeadDim;
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) {
        float v[32];
        if (ok) tmem_ld_32x32b_x32(t_lane + kTmemO + ch * 32, v);
        if (ok && row_ok) {
          float4* d4 = reinterpret_cast<float4*>(po + ch * 32);
#pragma unroll
          for (int x = 0; x < 8; ++x)
            d4[x] = make_float4(v[4 * x] * inv, v[4 * x + 1] * inv, v[4 * x + 2] * inv,
                                v[4 * x + 3] * inv);
        }
      }
      if (row_ok) p.ws_lse[slot] = (l_run > 0.f) ? m_run + __log2f(l_run) : -INFINITY;
      __threadfence();
      named_bar_sync(1, 128);
      if (m == 0) {
        int last = 0;
        if (*reinterpret_cast<volatile int*>(&bars->abort) == 0) {
          const int prev = atomicAdd(&p.ws_count[unit], 1);
          last = (prev == active - 1);
        }
        bars->last = last;
      }
      named_bar_sync(1, 128);
      if (*reinterpret_cast<volatile int*>(&bars->last)) {
        __threadfence();
        if (row_ok) {
          const long long base = unit * p.splits * kBlockM + m;
          float lmax = -INFINITY;
          for (int sp2 = 0; sp2 < active; ++sp2)
            lmax = fmaxf(lmax, __ldcg(p.ws_lse + base + sp2 * kBlockM));
          float acc[kHeadDim];
#pragma unroll
          for (int d = 0; d < kHeadDim; ++d) acc[d] = 0.f;
          float wsum = 0.f;
          for (int sp2 = 0; sp2 < active; ++sp2) {
            const float lse = __ldcg(p.ws_lse + base + sp2 * kBlockM);
            const float w = (lse == -INFINITY) ? 0.f : fast_exp2(lse - lmax);
            wsum += w;
            const float4* src =
                reinterpret_cast<const float4*>(p.ws_o + (base + sp2 * kBlockM) * kHeadDim);
#pragma unroll
            for (int d4 = 0; d4 < kHeadDim / 4; ++d4) {
              const float4 o = __ldcg(src + d4);
              acc[4 * d4 + 0] = fmaf(w, o.x, acc[4 * d4 + 0]);
              acc[4 * d4 + 1] = fmaf(w, o.y, acc[4 * d4 + 1]);
              acc[4 * d4 + 2] = fmaf(w, o.z, acc[4 * d4 + 2]);
              acc[4 * d4 + 3] = fmaf(w, o.w, acc[4 * d4 + 3]);
            }
          }
          const float inv2 = 1.f / wsum;
          uint4* d4 = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(p.out) +
                                               (static_cast<long long>(row0 + r) * p.Hq + h) *
                                                   kHeadDim);
#pragma unroll
          for (int x = 0; x < kHeadDim / 8; ++x)
            d4[x] = make_uint4(pack_bf16(acc[8 * x + 0] * inv2, acc[8 * x + 1] * inv2),
                               pack_bf16(acc[8 * x + 2] * inv2, acc[8 * x + 3] * inv2),
                               pack_bf16(acc[8 * x + 4] * inv2, acc[8 * x + 5] * inv2),
                               pack_bf16(acc[8 * x + 6] * inv2, acc[8 * x + 7] * inv2));
        }
        if (m == 0) atomicExch(&p.ws_count[unit], 0);
      }
    }
  }

  // ---- teardown ----
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

size_t tc_smem_bytes() { return kSmemBytes; }

cudaError_t launch_slot_attn_tc(const CUtensorMap& map_q, const CUtensorMap& map_k,
                                const CUtensorMap& map_v, const TcParams& p,
                                cudaStream_t stream) {
  static thread_local int configured_device = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured_device != dev) {
    e = cudaFuncSetAttribute(slot_attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kSmemBytes));
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  dim3 grid(p.m_tiles, p.splits, p.B * p.Hkv);
  slot_attn_tc_kernel<<<grid, kThreads, kSmemBytes, stream>>>(map_q, map_k, map_v, p);
  return cudaGetLastError();
}

}  // namespace zarya
