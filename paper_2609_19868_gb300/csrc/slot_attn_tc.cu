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
//     swizzle; paged caches use one box per page), K and V on separate rings
//     with separate producer warps;
//   * two softmax warpgroups take alternate key tiles. Each owns an S buffer
//     and an O accumulator in TMEM; P (bf16) is written back over the first
//     half of its S buffer and P*V takes it straight from TMEM, so shared
//     memory holds only Q and the K/V rings (3 stages each). The softmax of
//     tile i+1 runs while tile i's P*V and tile i+2's Q*K^T run. The two
//     partial results (O_b, running max m_b, sum l_b) are merged per row at
//     the end;
//   * S = Q K^T and O += P V are tcgen05.mma ops issued by one thread, in the
//     order Q*K^T(0), Q*K^T(1), then P*V(i), Q*K^T(i+2) for each i: the
//     tensor pipe runs one thread's MMAs in issue order, so P*V(i) has read
//     P(i) before Q*K^T(i+2) overwrites that buffer, and a completed Q*K^T(i)
//     implies P*V(i-2) is complete too. The softmax reads S with tcgen05.ld,
//     applies the mask from indices, and runs the online softmax (exp2 on the
//     MUFU, rescaling O only when the running maximum grows by more than 2^8);
//   * when the key range is split across CTAs, the splits of a tile form a
//     thread-block cluster (up to 3): splits > 0 push their partial into
//     split 0's shared memory with a bulk copy and split 0 merges in split
//     order; more splits merge through the workspace:
//     O = sum_s 2^(lse_s - M) O_s / sum_s 2^(lse_s - M),  M = max_s lse_s.
//
// Warp roles (384 threads): warp 0 K producer (and Q), warp 1 MMA issuer
// (one elected lane issues),
// warp 2 V producer, warp 3 TMEM allocator, warps 4-7 softmax group 0 (even
// tiles), warps 8-11 softmax group 1 (odd tiles). Warp w reads TMEM lanes
// 32*(w%4) .. +31, i.e. the packed rows of that range.
//
// Every mbarrier wait is bounded (p.wait_ns of global time, 2 s unless the
// caller sets another limit); a wait that gives up records
// ZARYA_DEVERR_TIMEOUT, raises a CTA-wide abort flag and the CTA unwinds
// (draining its own copies and MMAs, freeing TMEM).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "internal.cuh"
#include "ptx.cuh"

namespace zarya {
namespace {

constexpr int kThreads = 384;
constexpr int kSoftmaxWarps = 8;   // warps 4..11: two softmax warpgroups
// Tiles of K and of V warmed in L2 before the grid dependency wait (all CTAs'
// first tiles then land before the rest of the ring prefill).
constexpr int kPrefetchTiles = 2;
constexpr int kStagesK = 3;
constexpr int kStagesV = 3;
constexpr uint32_t kHalfBytes = kBlockN * 64 * 2;   // 128 rows x 128 B
constexpr uint32_t kTileBytes = 2 * kHalfBytes;     // 32 KB (128 x 128 bf16)
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kOffQ + kTileBytes;
constexpr uint32_t kOffV = kOffK + kStagesK * kTileBytes;
constexpr uint32_t kOffBar = kOffV + kStagesV * kTileBytes;
constexpr uint32_t kTmemCols = 512;  // S0/P0 [0,128) S1/P1 [128,256) O0 [256,384) O1 [384,512)
constexpr uint32_t kTmemO = 256;
constexpr uint64_t kDrainNs = 100000000ull;  // 100 ms

struct Bars {
  uint64_t q_full;
  uint64_t k_full[kStagesK];
  uint64_t k_empty[kStagesK];
  uint64_t v_full[kStagesV];
  uint64_t v_empty[kStagesV];
  uint64_t s_full[2];
  uint64_t p_full[2];
  uint64_t o_done[2];   // o_done[i & 1], phase i >> 1: P*V(i) has completed
  uint64_t drain;
  uint64_t kfree;   // this CTA's last Q*K^T has completed: its K ring is idle
  uint64_t staged;  // staged attention: the block rows this CTA reads are in the cache
  uint64_t stage_issued;  // staged attention: the first round of staging loads is issued
  uint64_t ready;   // cluster merge: every partial row this CTA owns has landed
  uint64_t go;      // cluster merge: every other split's K ring is free to receive
  uint64_t stall;   // never completed: the debug stall waits on it until its limit
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

// max(a, b, c) in one instruction (the three-input form of max.f32).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Row maximum of 64 scores: four chains of sixteen, 34 max instructions.
__device__ __forceinline__ float max64(const float (&s)[64]) {
  float m4[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    float a = fmax3(s[k], s[k + 4], s[k + 8]);
#pragma unroll
    for (int x = 12; x < 60; x += 8) a = fmax3(a, s[x + k], s[x + 4 + k]);
    m4[k] = fmaxf(a, s[60 + k]);
  }
  return fmax3(fmaxf(m4[0], m4[1]), m4[2], m4[3]);
}

// The softmax numerators of one row over 64 score columns, s[c] → 2^(s[c] *
// sl2 - m), packed as 32 bf16 pairs into pk; returns their fp32 sum.  The
// exponent arguments and the four running sums use the paired fp32
// instructions.  Each half rounds exactly as the scalar fmaf / add would, so
// the result is the scalar loop's bit for bit, with half the issue slots.
__device__ __forceinline__ float exp_pack_row(const float* s, float sl2, float m,
                                              float pk[32]) {
  const float2 k = make_float2(sl2, sl2), nm = make_float2(-m, -m);
  float2 r01 = make_float2(0.f, 0.f), r23 = make_float2(0.f, 0.f);
#pragma unroll
  for (int x = 0; x < 32; x += 2) {
    const int c = 2 * x;
    const float2 a01 = __ffma2_rn(make_float2(s[c + 0], s[c + 1]), k, nm);
    const float2 a23 = __ffma2_rn(make_float2(s[c + 2], s[c + 3]), k, nm);
    const float2 e01 = make_float2(fast_exp2(a01.x), fast_exp2(a01.y));
    const float2 e23 = make_float2(fast_exp2(a23.x), fast_exp2(a23.y));
    r01 = __fadd2_rn(r01, e01);
    r23 = __fadd2_rn(r23, e23);
    pk[x] = __uint_as_float(pack_bf16(e01.x, e01.y));
    pk[x + 1] = __uint_as_float(pack_bf16(e23.x, e23.y));
  }
  return (r01.x + r01.y) + (r23.x + r23.y);
}

__device__ __forceinline__ void named_bar_sync(int id, int n) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

__device__ __forceinline__ void named_bar_arrive(int id, int n) {
  asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// Named barrier that also ANDs a flag over its n threads (every participant
// arrives whatever its flag, so the group leaves together).
__device__ __forceinline__ bool named_bar_and(int id, int n, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %3, 0;\n\t"
      "bar.red.and.pred po, %1, %2, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(r)
      : "r"(id), "r"(n), "r"(v ? 1u : 0u)
      : "memory");
  return r != 0;
}

// Named barriers (barrier 0 is __syncthreads): 1 joins the 256 softmax
// threads, 2-5 one quadrant's warp of each softmax group, 7 publishes the
// entry set-up to the other ten warps.
constexpr int kBarSoftmax = 1;
constexpr int kBarSetup = 7;

template <class BarsT>
__device__ __forceinline__ void set_abort(BarsT* bars, int* err, int code) {
  record_error(err, code);
  *reinterpret_cast<volatile int*>(&bars->abort) = 1;
}

// Bounded wait (p.wait_ns of global time) for a phase of a barrier of this CTA.
template <class BarsT>
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, BarsT* bars,
                                         const TcParams& p) {
  if (mbar_wait(bar, parity, p.wait_ns, &bars->abort)) return true;
  set_abort(bars, p.err, ZARYA_DEVERR_TIMEOUT);
  return false;
}

// Cluster merge layout. Packed rows are handled in quadrants of 32 (one warp
// of each softmax group); quadrant q is finished by split q % active. A
// quadrant's partial (32 rows x 128 fp32 columns, 16 KB, plus 32 lse values)
// is staged by each other split in its idle V ring and pushed with one bulk
// copy into the owner's idle K ring, slot (sender's rank among the owner's
// peers, q / active).
constexpr uint32_t kQuadBytes = 32 * kHeadDim * 4;
constexpr uint32_t kQuadLseBytes = 32 * 4;
constexpr uint32_t kRxLse = 64 * 1024;   // lse slots follow the data slots

__device__ __forceinline__ uint32_t cmerge_rx_bytes(int n_rows, int active, int split) {
  const int nq = (n_rows + 31) >> 5;
  int owned = 0;
  for (int q = split; q < nq; q += active) ++owned;
  return static_cast<uint32_t>((active - 1) * owned) * (kQuadBytes + kQuadLseBytes);
}

// Swizzled byte offset of 16-byte chunk `chunk` (0..31) of row `L` (0..31) of
// a quadrant: lanes L of a warp touch distinct chunks of their rows.
__device__ __forceinline__ uint32_t quad_chunk(int L, int chunk) {
  return static_cast<uint32_t>(L) * 512u + (static_cast<uint32_t>(chunk ^ L) << 4);
}

__device__ __forceinline__ void st_shared_f4(uint32_t a, float x, float y, float z, float w) {
  asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(a), "f"(x), "f"(y), "f"(z),
               "f"(w)
               : "memory");
}

__device__ __forceinline__ float4 ld_shared_f4(uint32_t a) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(a)
               : "memory");
  return v;
}

__device__ __forceinline__ float ld_shared_f32(uint32_t a) {
  float v;
  asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
  return v;
}

// Owner side of the cluster merge for one row: this split's normalised
// partial o (64 columns of group grp) and the A - 1 partials received from the
// other splits, O = sum_s 2^(lse_s - M) O_s / sum_s 2^(lse_s - M), stored as
// bf16. rx / rx_lse address the first peer slot of this row (shared::cta).
template <int A>
__device__ __forceinline__ void cluster_merge_store(const float (&o)[64], float lse_own,
                                                    uint32_t rx, uint32_t rx_lse, int L, int grp,
                                                    __nv_bfloat16* out_row) {
  float lp[A - 1];
  float M = lse_own;
#pragma unroll
  for (int k = 0; k < A - 1; ++k) {
    lp[k] = ld_shared_f32(rx_lse + k * 2 * kQuadLseBytes);
    M = fmaxf(M, lp[k]);
  }
  float wo = lse_own == -INFINITY ? 0.f : fast_exp2(lse_own - M);
  float wp[A - 1];
  float S = wo;
#pragma unroll
  for (int k = 0; k < A - 1; ++k) {
    wp[k] = lp[k] == -INFINITY ? 0.f : fast_exp2(lp[k] - M);
    S += wp[k];
  }
  const float inv = S > 0.f ? 1.f / S : 0.f;
  wo *= inv;
#pragma unroll
  for (int k = 0; k < A - 1; ++k) wp[k] *= inv;
  uint4* d4 = reinterpret_cast<uint4*>(out_row);
#pragma unroll
  for (int x = 0; x < 8; ++x) {
    float r[8];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int c = 2 * x + h;
      float4 acc = make_float4(wo * o[4 * c], wo * o[4 * c + 1], wo * o[4 * c + 2], wo * o[4 * c + 3]);
#pragma unroll
      for (int k = 0; k < A - 1; ++k) {
        const float4 v = ld_shared_f4(rx + k * 2 * kQuadBytes + quad_chunk(L, grp * 16 + c) -
                                      static_cast<uint32_t>(L) * 512u);
        acc.x = fmaf(wp[k], v.x, acc.x);
        acc.y = fmaf(wp[k], v.y, acc.y);
        acc.z = fmaf(wp[k], v.z, acc.z);
        acc.w = fmaf(wp[k], v.w, acc.w);
      }
      r[4 * h] = acc.x;
      r[4 * h + 1] = acc.y;
      r[4 * h + 2] = acc.z;
      r[4 * h + 3] = acc.w;
    }
    d4[x] = make_uint4(pack_bf16(r[0], r[1]), pack_bf16(r[2], r[3]), pack_bf16(r[4], r[5]),
                       pack_bf16(r[6], r[7]));
  }
}

// Bounded wait (acquire at cluster scope) for a phase completed by other CTAs
// of the cluster.
__device__ __forceinline__ bool wait_bar_cluster(uint64_t* bar, uint32_t parity, Bars* bars,
                                                 const TcParams& p) {
  if (mbar_wait_cluster(bar, parity, p.wait_ns, &bars->abort)) return true;
  set_abort(bars, p.err, ZARYA_DEVERR_TIMEOUT);
  return false;
}

// Staged attention: warp 3 (idle until the merge) copies the block rows
// [i_lo, i_hi) of sequence b, KV head kvh, of K and V from k_new / v_new
// ([total_rows, Hkv, D]) to cache positions P + i, with kRound 16-byte
// vectors of each tensor per lane in flight per round, then fences the writes
// against the async proxy; the producers wait on `staged` before loading the
// first tile that holds one of these rows.
// Staged attention: the block rows this CTA reads are copied from k_new /
// v_new into the cache by the eight softmax warps (idle until the first score
// tile). The loads of the first round are issued before the producers' first
// tensor copies (16-byte loads issued behind this SM's tensor streams return
// only when those streams end); the stores, any further rounds and the proxy
// fence follow the set-up barrier.
struct GroupStager {
  static constexpr int kVec = kHeadDim * 2 / 16;   // 16-byte vectors per (token, head) row
  static constexpr int kThreads = kSoftmaxWarps * 32;
  static constexpr int kRound = 2;                 // vectors of K and of V per thread per round
  uint4 vk[kRound], vv[kRound];
  long long d[kRound];

  __device__ __forceinline__ void load(const TcParams& p, int b, int kvh, int row0, int P,
                                       int i_lo, int i_hi, int t, int base) {
    const uint4* kn = static_cast<const uint4*>(p.k_new);
    const uint4* vn = static_cast<const uint4*>(p.v_new);
    const int n = (i_hi - i_lo) * kVec;
#pragma unroll
    for (int u = 0; u < kRound; ++u) {
      const int idx = base + u * kThreads + t;
      d[u] = -1;
      if (idx < n) {
        const int i = i_lo + idx / kVec;
        const int c = idx % kVec;
        const int tok = P + i;
        long long tr = -1;
        if (p.page_size == 0) {
          tr = static_cast<long long>(b) * p.capacity + tok;
        } else {
          const int page =
              p.page_table[static_cast<long long>(b) * p.max_pages + tok / p.page_size];
          if (page < 0 || page >= p.n_pages) record_error(p.err, ZARYA_DEVERR_PAGE_ID);
          else tr = static_cast<long long>(page) * p.page_size + tok % p.page_size;
        }
        if (tr >= 0) {
          const long long sidx = (static_cast<long long>(row0 + i) * p.Hkv + kvh) * kVec + c;
          vk[u] = __ldg(kn + sidx);
          vv[u] = __ldg(vn + sidx);
          d[u] = (tr * p.Hkv + kvh) * kVec + c;
        }
      }
    }
  }

  __device__ __forceinline__ void store(const TcParams& p) {
    uint4* kc = static_cast<uint4*>(p.k_cache);
    uint4* vc = static_cast<uint4*>(p.v_cache);
#pragma unroll
    for (int u = 0; u < kRound; ++u) {
      if (d[u] >= 0) {
        kc[d[u]] = vk[u];
        vc[d[u]] = vv[u];
      }
    }
  }

  // Stores the first round, copies the rest, and makes the writes visible to
  // the tensor copies that will read them.
  __device__ __forceinline__ void finish(const TcParams& p, int b, int kvh, int row0, int P,
                                         int i_lo, int i_hi, int t) {
    store(p);
    const int n = (i_hi - i_lo) * kVec;
    for (int base = kRound * kThreads; base < n; base += kRound * kThreads) {
      load(p, b, kvh, row0, P, i_lo, i_hi, t, base);
      store(p);
    }
    asm volatile("fence.proxy.async.global;" ::: "memory");
  }
};

// One producer warp streams one of K or V through its ring.
// One producer warp streams one of K or V through its ring: tiles
// [i_begin, i_end) of this CTA's range, `issued` counting the tiles whose
// copies are in flight. Returns false (the CTA aborts) on a bad page id or a
// timed-out wait.
template <class BarsT>
__device__ __forceinline__ bool produce_range(const CUtensorMap* map, uint64_t* full,
                                              uint64_t* empty, int stages, uint32_t ring,
                                              const TcParams& p, BarsT* bars, int b, int kvh,
                                              int t_begin, int i_begin, int i_end, int kv_end,
                                              int lane, int t_stage, int& issued) {
  const bool paged = p.page_size > 0;
  const int ppt = paged ? kBlockN / p.page_size : 0;   // pages per tile
  const uint32_t page_bytes = paged ? static_cast<uint32_t>(p.page_size) * 256u : 0u;
  // Lane l's page of tile i (-1 when the tile has no such page). The page ids
  // of the next tile are read one tile ahead, before this tile's waits, so
  // their latency hides behind the ring instead of delaying the copies.
  auto page_of = [&](int i) -> int {
    const int lp = (t_begin + i) * ppt + lane;
    if (lane >= ppt || lp * p.page_size >= kv_end) return -1;
    return p.page_table[static_cast<long long>(b) * p.max_pages + lp];
  };
  int page_next = (paged && i_begin < i_end) ? page_of(i_begin) : -1;
  for (int i = i_begin; i < i_end; ++i) {
    const int t = t_begin + i;
    int page = -1;
    uint32_t bytes = kTileBytes;
    if (paged) {
      page = page_next;
      if (i + 1 < i_end) page_next = page_of(i + 1);
    }
    if (t == t_stage && !wait_bar(&bars->staged, 0, bars, p)) return false;
    if (paged) {
      const int lp = t * ppt + lane;
      const bool want = lane < ppt && lp * p.page_size < kv_end;
      const bool bad = want && (page < 0 || page >= p.n_pages);
      if (__any_sync(0xffffffffu, bad)) {
        if (lane == 0) set_abort(bars, p.err, ZARYA_DEVERR_PAGE_ID);
        return false;
      }
      bytes = page_bytes * __popc(__ballot_sync(0xffffffffu, want));
    }
    const int s = i % stages;
    bool w = true;
    if (lane == 0) {
      w = wait_bar(&empty[s], ((i / stages) & 1) ^ 1, bars, p);
      if (w) mbar_arrive_expect_tx(&full[s], bytes);
    }
    if (!__shfl_sync(0xffffffffu, w, 0)) return false;
    issued = i + 1;
    const uint32_t dst = ring + s * kTileBytes;
    if (!paged) {
      if (lane == 0) {
        tma_load_4d(dst, map, &full[s], 0, kvh, t * kBlockN, b);
        tma_load_4d(dst + kHalfBytes, map, &full[s], 64, kvh, t * kBlockN, b);
      }
    } else if (page >= 0) {
      const uint32_t o = lane * p.page_size * 128;
      tma_load_4d(dst + o, map, &full[s], 0, kvh, 0, page);
      tma_load_4d(dst + kHalfBytes + o, map, &full[s], 64, kvh, 0, page);
    }
  }
  return true;
}

// L2 prefetch of the first kPrefetchTiles tiles of this CTA's key range (and of its
// Q tile when map_q is given), from a reading of the sequence's lengths that
// may be stale; nothing is prefetched when that reading is out of range.
__device__ __forceinline__ void prefetch_first_tiles(const CUtensorMap* map_kv,
                                                     const CUtensorMap* map_q, const TcParams& p,
                                                     int b, int kvh, int mt, int split) {
  const int P = ld_relaxed_gpu(p.cache_lens + b);
  const long long R64 = static_cast<long long>(ld_relaxed_gpu(p.n_slots + b)) *
                        ld_relaxed_gpu(p.slot_len + b);
  const int mode = ld_relaxed_gpu(p.mask_mode + b);
  const int row0 = ld_relaxed_gpu(p.q_row_offsets + b);
  if (P < 0 || R64 < 1 || R64 > p.max_rows || P + R64 > p.capacity) return;
  const int R = static_cast<int>(R64);
  const int rows_per_tile = kBlockM / p.g;
  const int r0 = mt * rows_per_tile;
  if (r0 >= R) return;
  const int r_hi = min(r0 + rows_per_tile, R) - 1;
  const int kv_end = mode == ZARYA_MASK_BIDIR_BLOCK ? P + R : P + r_hi + 1;
  const int n_tiles = (kv_end + kBlockN - 1) / kBlockN;
  const int per_split = max(1, (n_tiles + p.splits - 1) / p.splits);
  const int t_begin = split * per_split;
  const int t_end = min(n_tiles, t_begin + min(per_split, kPrefetchTiles));
  for (int t = t_begin; t < t_end; ++t) {
    tma_prefetch_l2_4d(map_kv, 0, kvh, t * kBlockN, b);
    tma_prefetch_l2_4d(map_kv, 64, kvh, t * kBlockN, b);
  }
  if (map_q != nullptr && row0 >= 0 && row0 + r0 < p.total_rows) {
    tma_prefetch_l2_3d(map_q, 0, kvh * p.g, row0 + r0);
    tma_prefetch_l2_3d(map_q, 64, kvh * p.g, row0 + r0);
  }
}

// After a failed produce_range: let this CTA's own copies land before the CTA
// (and its shared memory) goes away.
__device__ __forceinline__ void drain_ring(uint64_t* full, int stages, int issued, int lane) {
  if (lane == 0)
    for (int i = max(0, issued - stages); i < issued; ++i)
      mbar_wait(&full[i % stages], (i / stages) & 1, kDrainNs, nullptr);
}

// The work tile of the CTA at linear position pos under the schedule: item
// perm[pos / Hkv] (sequence item / items, tile item % items), KV head
// pos % Hkv. Returns false for an item outside [0, B x items).
__device__ __forceinline__ bool scheduled_tile(const TcParams& p, int item, int pos, int& b,
                                               int& kvh, int& t) {
  if (item < 0 || item >= p.B * p.items) return false;
  b = item / p.items;
  t = item - b * p.items;
  kvh = pos % p.Hkv;
  return true;
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

  // ---- set-up that needs no input (overlaps the previous kernel's tail) ----
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_q);
    tma_prefetch_map(&map_k);
    tma_prefetch_map(&map_v);
  }
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
      mbar_init(&bars->p_full[s], 8);   // every softmax warp, each tile
    }
    mbar_init(&bars->o_done[0], 1);
    mbar_init(&bars->o_done[1], 1);
    mbar_init(&bars->drain, 1);
    mbar_init(&bars->kfree, 1);
    mbar_init(&bars->staged, kSoftmaxWarps);
    mbar_init(&bars->stage_issued, kSoftmaxWarps);
    mbar_init(&bars->stall, 1);
    bars->abort = 0;
    bars->last = 0;
    fence_mbar_init();
  }
  // Every barrier is initialised before any thread touches one. The softmax
  // warps signal stage_issued before the CTA-wide set-up barrier below, so
  // without this barrier their arrive could land before thread 0's
  // initialisation and be lost, and the producers' wait for it would run out.
  // No copy is in flight yet, so nothing holds a thread here.
  __syncthreads();
  if (warp == 3) {
    tmem_alloc(&bars->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  // The producer warps load before the CTA-wide set-up barrier (a thread
  // with tensor copies in flight waits for them at a barrier): they arrive,
  // without waiting, on the set-up barrier the other ten warps wait on.
  if (warp == 0 || warp == 2) named_bar_arrive(kBarSetup, kThreads);
  // Before waiting for the kernel launched before this one, warm L2 with Q
  // and the first tiles of this split's K / V. L2 is the point of coherence,
  // so a prefetch cannot hand stale data to the loads made after the wait;
  // the lengths read here (that kernel may still be writing them) only steer
  // which lines are warmed. Contiguous caches only.
  if ((warp == 0 || warp == 2) && lane == 0 && p.page_size == 0)
    prefetch_first_tiles(warp == 0 ? &map_k : &map_v, warp == 0 ? &map_q : nullptr, p, b, kvh,
                         mt, split);
  // Inputs may be written by the kernel launched before this one.
  grid_dependency_wait();

  // ---- per-sequence geometry (uniform over the CTA) ----
  const int P = p.cache_lens[b];
  // R_b = S_b * L_b, clamped so that an absurd product reads as invalid below
  const long long R64 = static_cast<long long>(p.n_slots[b]) * p.slot_len[b];
  const int R = R64 > p.max_rows ? p.max_rows + 1 : static_cast<int>(R64);
  const int mode = p.mask_mode[b];
  const int row0 = p.q_row_offsets[b];
  const int row_end = p.q_row_offsets[b + 1];
  int code = 0;
  if (mode != ZARYA_MASK_BIDIR_BLOCK && mode != ZARYA_MASK_SLOT_CAUSAL &&
      mode != ZARYA_MASK_SLOT_INDEPENDENT)
    code = ZARYA_DEVERR_MASK_MODE;
  else if (p.n_slots[b] < 1 || p.slot_len[b] < 1 || R > p.max_rows || row_end - row0 != R ||
           row0 < 0 || row_end > p.total_rows)
    code = ZARYA_DEVERR_ROWS;
  else if (P < 0 || static_cast<long long>(P) + R > p.capacity) code = ZARYA_DEVERR_CAPACITY;
  const int rows_per_tile = kBlockM / p.g;
  const int r0 = mt * rows_per_tile;
  const int r_hi = min(r0 + rows_per_tile, R) - 1;
  const int kv_end = (mode == ZARYA_MASK_BIDIR_BLOCK) ? P + R : P + r_hi + 1;
  const int n_tiles = (code != 0 || kv_end <= 0) ? 1 : (kv_end + kBlockN - 1) / kBlockN;
  const int per_split = max(1, (n_tiles + p.splits - 1) / p.splits);
  const int active = (n_tiles + per_split - 1) / per_split;
  const int t_begin = split * per_split;
  const int nt = min(n_tiles, t_begin + per_split) - t_begin;
  // Staged attention: the block rows this CTA reads, [st_lo, st_hi) relative to P.
  int st_lo = 0, st_hi = 0;
  if (p.k_new != nullptr && code == 0) {
    st_lo = max(P, t_begin * kBlockN) - P;
    st_hi = min(kv_end, (t_begin + nt) * kBlockN) - P;
  }

  // The splits of a cluster merge their partials through shared memory when
  // more than one of them has keys (Sec. 5.2 step 3 split over the key range).
  const bool cmerge = p.cluster != 0 && active > 1;
  if (threadIdx.x == 32) {
    mbar_init(&bars->go, cmerge ? active - 1 : 1);
    mbar_init(&bars->ready, 1);
    fence_mbar_init();
    // The bytes the other splits will push (their rows of the quadrants this
    // split finishes) are known here, so the barrier is armed before any peer
    // can start a copy.
    if (cmerge) {
      const int n_rows_v = min(kBlockM, (r_hi - r0 + 1) * p.g);
      mbar_arrive_expect_tx(&bars->ready, cmerge_rx_bytes(n_rows_v, active, split));
    }
  }
  // The cluster barrier orders every CTA's barrier initialisation (released by
  // fence.mbarrier_init) before any remote arrive; its wait is taken only
  // where a thread first needs it. Arriving before the producers issue their
  // first copies keeps the arrive from waiting on them.
  if (p.cluster) cluster_arrive_relaxed();

  // Producers issue Q and the first ring stages as soon as their own geometry
  // is known (contiguous caches; stopping before a tile that holds a staged
  // block row), before the CTA-wide barrier.
  const bool works = code == 0 && r0 < R && split < active;
  const int t_stage = st_hi > st_lo ? (P + st_lo) / kBlockN : -1;
  int pre = 0;   // tiles issued before the barrier by each producer
  if (works && p.page_size == 0) {
    pre = min(nt, kStagesK);
    if (t_stage >= 0) pre = min(pre, t_stage - t_begin);
  }
  int issued = 0;
  const bool stage_here = works && st_hi > st_lo;
  GroupStager stg;
  if (warp >= 4 && stage_here) {
    stg.load(p, b, kvh, row0, P, st_lo, st_hi, threadIdx.x - 128, 0);
    __syncwarp();
    if (lane == 0) mbar_arrive_relaxed(&bars->stage_issued);
  }
  if ((warp == 0 || warp == 2) && works) {
    if (stage_here) {
      // a timeout sets the abort flag; the ring loop below then returns early
      if (lane == 0) wait_bar(&bars->stage_issued, 0, bars, p);
      __syncwarp();
    }
    const bool is_k = warp == 0;
    if (is_k) {
      if (lane == 0) {
        mbar_arrive_expect_tx(&bars->q_full, kTileBytes);
        const uint32_t dq = smem_u32(smem + kOffQ);
        tma_load_3d(dq, &map_q, &bars->q_full, 0, kvh * p.g, row0 + r0);
        tma_load_3d(dq + kHalfBytes, &map_q, &bars->q_full, 64, kvh * p.g, row0 + r0);
      }
      produce_range(&map_k, bars->k_full, bars->k_empty, kStagesK, smem_u32(smem + kOffK), p,
                    bars, b, kvh, t_begin, 0, pre, kv_end, lane, t_stage, issued);
    } else {
      produce_range(&map_v, bars->v_full, bars->v_empty, kStagesV, smem_u32(smem + kOffV), p,
                    bars, b, kvh, t_begin, 0, pre, kv_end, lane, t_stage, issued);
    }
  }

  if (warp != 0 && warp != 2) {
    tc_fence_before();
    named_bar_sync(kBarSetup, kThreads);
    tc_fence_after();
  }
  // TMEM base address (warp 3 wrote it before the set-up barrier); the
  // producer warps never use it.
  const uint32_t tmem = (warp != 0 && warp != 2) ? bars->tmem_base : 0u;
  bool cwaited = false;
  bool mma_issued = false;   // the MMA warp issued at least one tcgen05.mma
  // Exits here are uniform over a cluster (its CTAs share the sequence and
  // M-tile and differ only in the split) or leave a split with no keys.
  if (!works) {
    if (code != 0 && mt == 0 && split == 0 && threadIdx.x == 0) record_error(p.err, code);
    grid_launch_dependents();
    if (p.cluster) cluster_wait();
    if (warp == 3) tmem_dealloc(tmem, kTmemCols);
    return;
  }

  if (warp < 4) {
    if (warp == 0) {
      // ======================= Q + K producer =======================
      // (Q and the first `pre` K tiles were issued before the CTA barrier.)
      if (!produce_range(&map_k, bars->k_full, bars->k_empty, kStagesK, smem_u32(smem + kOffK), p,
                         bars, b, kvh, t_begin, pre, nt, kv_end, lane, t_stage, issued))
        drain_ring(bars->k_full, kStagesK, issued, lane);
      if (lane == 0 && *reinterpret_cast<volatile int*>(&bars->abort) != 0)
        mbar_wait(&bars->q_full, 0, kDrainNs, nullptr);
    } else if (warp == 2) {
      // ======================= V producer =======================
      if (!produce_range(&map_v, bars->v_full, bars->v_empty, kStagesV, smem_u32(smem + kOffV), p,
                         bars, b, kvh, t_begin, pre, nt, kv_end, lane, t_stage, issued))
        drain_ring(bars->v_full, kStagesV, issued, lane);
    } else if (warp == 1) {
      // ======================= MMA issuer (one elected lane) =======================
      // The whole warp walks the issue loop (waits and descriptors are
      // warp-uniform); elect.sync picks the lane that issues MMAs and commits.
      bool ok = true;
      // Failure-path test: a wait that nothing completes runs out after
      // p.wait_ns and the CTA unwinds like after any other timeout.
      if (p.debug_stall) ok = wait_bar(&bars->stall, 0, bars, p);
      if (ok) ok = wait_bar(&bars->q_full, 0, bars, p);
      bool any_mma = false;
      tc_fence_after();
      const uint64_t q_desc0 = sdesc_sw128(smem_u32(smem + kOffQ), 16, 1024);
      const uint64_t q_desc1 = sdesc_sw128(smem_u32(smem + kOffQ + kHalfBytes), 16, 1024);
      const uint64_t k_desc0 = sdesc_sw128(smem_u32(smem + kOffK), 16, 1024);
      const uint64_t v_desc0 = sdesc_sw128(smem_u32(smem + kOffV), kHalfBytes, 1024);
      // descriptors count addresses in 16-byte units
      constexpr uint64_t kTileUnits = kTileBytes >> 4, kHalfUnits = kHalfBytes >> 4;
      auto issue_qk = [&](int i) -> bool {
        const int s = i % kStagesK;
        const int sb = i & 1;
        if (!wait_bar(&bars->k_full[s], (i / kStagesK) & 1, bars, p)) return false;
        tc_fence_after();
        const uint64_t kd = k_desc0 + s * kTileUnits;
  #pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t step = (kk >> 2) * kHalfUnits + (kk & 3) * 2;
          tc_mma_ss_elect(tmem + sb * 128, (kk < 4 ? q_desc0 : q_desc1) + (kk & 3) * 2,
                          kd + step, kIdescQK, kk > 0 ? 1u : 0u);
        }
        any_mma = true;
        tc_commit_elect(&bars->s_full[sb]);
        tc_commit_elect(&bars->k_empty[s]);
        if (cmerge && i == nt - 1) tc_commit_elect(&bars->kfree);
        return true;
      };
      auto issue_pv = [&](int i) -> bool {
        const int sv = i % kStagesV;
        const int sb = i & 1;
        const int j = i >> 1;
        if (!wait_bar(&bars->p_full[sb], j & 1, bars, p)) return false;
        if (!wait_bar(&bars->v_full[sv], (i / kStagesV) & 1, bars, p)) return false;
        tc_fence_after();
        const uint64_t vd = v_desc0 + sv * kTileUnits;
        // O_g += P_g(i) * V(i)[64g, 64g + 64): P_g is packed over columns
        // [64g, 64g + 32) of the tile's S buffer, 16 keys per 8 columns.
  #pragma unroll
        for (int g2 = 0; g2 < 2; ++g2)
  #pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_ts_elect(tmem + kTmemO + g2 * 128, tmem + sb * 128 + g2 * 64 + kk * 8,
                            vd + (g2 * 4 + kk) * 128, kIdescPV, (i > 0 || kk > 0) ? 1u : 0u);
        any_mma = true;
        tc_commit_elect(&bars->o_done[sb]);
        tc_commit_elect(&bars->v_empty[sv]);
        return true;
      };
      if (ok) ok = issue_qk(0);
      if (ok && nt > 1) ok = issue_qk(1);
      for (int i = 0; i < nt && ok; ++i) {
        if (!issue_pv(i)) { ok = false; break; }
        if (i + 2 < nt && !issue_qk(i + 2)) { ok = false; break; }
      }
      mma_issued = any_mma;
    } else if (warp == 3) {
      // ======================= cluster merge: K ring hand-off =======================
      // Once this CTA's last Q*K^T has completed no copy or MMA touches its K
      // ring again: tell the other splits they may write their rows into it.
      if (cmerge) {
        const bool freed = wait_bar(&bars->kfree, 0, bars, p);
        cluster_wait();
        cwaited = true;
        if (freed && lane == 0)
          for (int sp = 0; sp < active; ++sp)
            if (sp != split) mbar_arrive_remote(mapa_shared(smem_u32(&bars->go), sp));
      }
    }
  } else {
    // ======================= softmax + epilogue =======================
    // Both groups work on every key tile: group g takes its keys
    // [64g, 64g + 64) with a running max / sum of its own and accumulates
    // into O_g; the two partial softmaxes are merged per row at the end.
    // ---- staging of the block's own K/V (first round loaded before the rings) ----
    if (stage_here) {
      stg.finish(p, b, kvh, row0, P, st_lo, st_hi, threadIdx.x - 128);
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->staged);
    }
    const int grp = (warp - 4) >> 2;
    const int wq = warp & 3;
    const int m = wq * 32 + lane;                   // packed row = TMEM lane
    const int r = r0 + m / p.g;
    const int h = kvh * p.g + (m - (m / p.g) * p.g);
    const bool row_ok = r <= r_hi;
    const int limit = !row_ok ? kv_end : (mode == ZARYA_MASK_BIDIR_BLOCK ? P + R : P + r + 1);
    // slot-independent: the block rows of the earlier slots, [P, hide_hi)
    const int hide_hi =
        (row_ok && mode == ZARYA_MASK_SLOT_INDEPENDENT) ? P + (r / p.slot_len[b]) * p.slot_len[b] : P;
    const uint32_t t_row = tmem + (static_cast<uint32_t>(wq * 32) << 16);
    const uint32_t t_o = t_row + kTmemO + grp * 128;
    const float sl2 = p.scale_log2;
    float m_run = -INFINITY;  // running max, in scaled log2 units
    float l_run = 0.f;
    bool ok = true;


    for (int i = 0; i < nt; ++i) {
      const int sb = i & 1;
      const int c0 = (t_begin + i) * kBlockN + grp * 64;   // first key of this half
      const uint32_t t_s = t_row + sb * 128 + grp * 64;
      if (ok) ok = wait_bar(&bars->s_full[sb], (i >> 1) & 1, bars, p);
      if (!__all_sync(0xffffffffu, ok)) { ok = false; break; }
      tc_fence_after();
      float s[64];
      tmem_ld_32x32b_x64(t_s, s);

      if (c0 + 64 > limit) {
#pragma unroll
        for (int x = 0; x < 64; ++x)
          if (c0 + x >= limit) s[x] = -INFINITY;
      }
      if (hide_hi > P && c0 < hide_hi && c0 + 64 > P) {
#pragma unroll
        for (int x = 0; x < 64; ++x)
          if (c0 + x >= P && c0 + x < hide_hi) s[x] = -INFINITY;
      }
      const float m_new = fmaxf(m_run, max64(s) * sl2);
      const bool need = m_new > m_run + 8.0f;
      const bool warp_need = __any_sync(0xffffffffu, need);
      float alpha = 1.f;
      if (warp_need) {
        alpha = (m_run == -INFINITY) ? 0.f : fast_exp2(m_run - m_new);
        m_run = m_new;
        l_run *= alpha;
      }
      const float m_use = (m_run == -INFINITY) ? 0.f : m_run;

      // Rescaling O_g must wait for P*V(i-1), the last MMA that wrote it.
      // S(i) complete implies P*V(i-2) complete (issued before Q*K^T(i)), so
      // this parity wait on o_done[(i-1) & 1] cannot alias an older phase.
      if (warp_need && i > 0) {
        if (ok) ok = wait_bar(&bars->o_done[(i - 1) & 1], ((i - 1) >> 1) & 1, bars, p);
        tc_fence_after();
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          float v[32];
          const uint32_t a = t_o + ch * 32;
          tmem_ld_32x32b_x32(a, v);
#pragma unroll
          for (int x = 0; x < 32; ++x) v[x] *= alpha;
          tmem_st_32x32b_x32(a, v);
        }
      }
      // Keys at or past kv_end in the last tile: their V rows (stale smem,
      // unloaded pages or another sequence's cache) must be exact zeros, or a
      // NaN there would poison P*V even with P = 0. Each group clears the
      // rows of its own half.
      if (c0 + 64 > kv_end) {
        const int sv = i % kStagesV;
        if (ok) ok = wait_bar(&bars->v_full[sv], (i / kStagesV) & 1, bars, p);
        const int key = grp * 64 + (m & 63);
        if (ok && m < 64 && c0 + (m & 63) >= kv_end) {
          uint8_t* vrow = smem + kOffV + sv * kTileBytes + (key >> 3) * 1024 + (key & 7) * 128;
          const uint4 z = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
          for (int x = 0; x < 8; ++x) {
            reinterpret_cast<uint4*>(vrow)[x] = z;
            reinterpret_cast<uint4*>(vrow + kHalfBytes)[x] = z;
          }
        }
        // the zeros are generic-proxy writes; P*V reads V through the async proxy
        fence_proxy_async_smem();
      }
      // P = 2^(s * scale * log2 e - m) as packed bf16 pairs over the first 32
      // columns of this group's half of the S buffer (S is in registers).
      float pk[32];
      l_run += exp_pack_row(s, sl2, m_use, pk);
      tmem_st_32x32b_x32(t_s, pk);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->p_full[sb]);
    }

    // ---- epilogue: merge the two groups' partial results per row ----
    // Each group has seen the last S, so no Q*K^T reads Q any more: the Q
    // buffer carries the (max, sum) exchange between the groups, done while
    // the last P*V still runs.
    float* xch = reinterpret_cast<float*>(smem + kOffQ + grp * 1024);
    xch[m] = m_run;
    xch[128 + m] = l_run;
    named_bar_sync(kBarSoftmax, 256);
    const float* x0 = reinterpret_cast<const float*>(smem + kOffQ);
    const float* x1 = reinterpret_cast<const float*>(smem + kOffQ + 1024);
    const float mA = x0[m], lA = x0[128 + m];
    const float mB = x1[m], lB = x1[128 + m];
    const float mT = fmaxf(mA, mB);
    const float aA = (mA == -INFINITY) ? 0.f : fast_exp2(mA - mT);
    const float aB = (mB == -INFINITY) ? 0.f : fast_exp2(mB - mT);
    const float lT = aA * lA + aB * lB;
    const float inv = (lT > 0.f) ? 1.f / lT : 0.f;
    const float wA = aA * inv, wB = aB * inv;
    const long long unit = static_cast<long long>(bh) * p.m_tiles + mt;
    const int col0 = grp * 64;   // group g finishes columns [64g, 64g + 64)
    grid_launch_dependents();
    // The cluster barrier's wait (needed before the merge's first remote
    // access) is taken here, while the last P*V still runs.
    if (p.cluster) {
      cluster_wait();
      cwaited = true;
    }
    // The last P*V completes after every other MMA of the CTA; P*V(nt-3) is
    // known complete, so the parity wait cannot alias an older phase.
    if (ok) ok = wait_bar(&bars->o_done[(nt - 1) & 1], ((nt - 1) >> 1) & 1, bars, p);
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();

    // This CTA's result for its 64 columns of row m, normalised: O_0's
    // columns, then O_1's, one tensor-memory load (and wait) each.
    float o[64];
    if (ok) {
      tmem_ld_32x32b_x64(t_row + kTmemO + col0, o);
      float vb[64];
      tmem_ld_32x32b_x64(t_row + kTmemO + 128 + col0, vb);
#pragma unroll
      for (int x = 0; x < 64; ++x) o[x] = wA * o[x] + wB * vb[x];
    } else {
#pragma unroll
      for (int x = 0; x < 64; ++x) o[x] = 0.f;
    }
    __nv_bfloat16* out_row = reinterpret_cast<__nv_bfloat16*>(p.out) +
                             (static_cast<long long>(row0 + r) * p.Hq + h) * kHeadDim + col0;
    auto store_out = [&](const float (&v)[64], float scale) {
      uint4* d4 = reinterpret_cast<uint4*>(out_row);
#pragma unroll
      for (int x = 0; x < 8; ++x)
        d4[x] = make_uint4(pack_bf16(v[8 * x + 0] * scale, v[8 * x + 1] * scale),
                           pack_bf16(v[8 * x + 2] * scale, v[8 * x + 3] * scale),
                           pack_bf16(v[8 * x + 4] * scale, v[8 * x + 5] * scale),
                           pack_bf16(v[8 * x + 6] * scale, v[8 * x + 7] * scale));
    };
    if (active == 1) {
      if (ok && row_ok) store_out(o, 1.f);
    } else if (p.cluster) {
      // Split key range, the splits of this tile in one cluster (at most 3).
      // Each quadrant of 32 packed rows is finished by split q % active; the
      // other splits stage their normalised partial of it (O_s, lse_s) in
      // their idle V ring and, once the owner's K ring is idle (its `go`),
      // push it there with one bulk copy that completes on the owner's
      // `ready`. The owner merges
      //   O = sum_s 2^(lse_s - M) O_s / sum_s 2^(lse_s - M).
      const float lse_own = (lT > 0.f) ? mT + __log2f(lT) : -INFINITY;
      const int n_rows = min(kBlockM, (r_hi - r0 + 1) * p.g);   // valid packed rows
      const int q = wq;                                          // this warp's quadrant
      const int owner = q % active;
      const uint32_t sbase = smem_u32(smem);
      if (q * 32 < n_rows && owner != split) {
        const uint32_t stage = sbase + kOffV + q * kQuadBytes;
        const uint32_t stage_lse = sbase + kOffV + kRxLse + q * kQuadLseBytes;
#pragma unroll
        for (int c = 0; c < 16; ++c)
          st_shared_f4(stage + quad_chunk(lane, grp * 16 + c), o[4 * c], o[4 * c + 1], o[4 * c + 2],
                       o[4 * c + 3]);
        if (grp == 0)
          asm volatile("st.shared.f32 [%0], %1;" ::"r"(stage_lse + lane * 4), "f"(lse_own)
                       : "memory");
        fence_proxy_async_smem();   // the bulk copy reads through the async proxy
        named_bar_sync(2 + q, 64);  // this quadrant's warp of each group
        if (grp == 0 && lane == 0) {
          if (wait_bar_cluster(&bars->go, 0, bars, p)) {
            const int slot = (split < owner ? split : split - 1) * 2 + q / active;
            const uint32_t rbar = mapa_shared(smem_u32(&bars->ready), owner);
            bulk_copy_to_cluster(mapa_shared(sbase + kOffK + slot * kQuadBytes, owner), stage,
                                 kQuadBytes, rbar);
            bulk_copy_to_cluster(mapa_shared(sbase + kOffK + kRxLse + slot * kQuadLseBytes, owner),
                                 stage_lse, kQuadLseBytes, rbar);
            bulk_commit_and_wait_read();   // this CTA's smem must outlive the reads
          }
        }
      } else if (q * 32 < n_rows) {
        const bool got = wait_bar_cluster(&bars->ready, 0, bars, p);
        if (got && ok && row_ok) {
          const int j = q / active;
          const uint32_t rx = sbase + kOffK + j * kQuadBytes + lane * 512u;
          const uint32_t rx_lse = sbase + kOffK + kRxLse + j * kQuadLseBytes + lane * 4u;
          if (active == 2)
            cluster_merge_store<2>(o, lse_own, rx, rx_lse, lane, grp, out_row);
          else
            cluster_merge_store<3>(o, lse_own, rx, rx_lse, lane, grp, out_row);
        }
      }
    } else {
      // Split key range beyond a cluster: every split writes its partial to
      // the workspace, takes a ticket, and the last one merges all of them in
      // split order (so the result does not depend on the arrival order).
      const float lse_own = (lT > 0.f) ? mT + __log2f(lT) : -INFINITY;
      const long long own = (unit * p.splits + split) * kBlockM + m;
      if (ok && row_ok) {
        float4* d4 = reinterpret_cast<float4*>(p.ws_o + own * kHeadDim + col0);
#pragma unroll
        for (int x = 0; x < 16; ++x)
          d4[x] = make_float4(o[4 * x], o[4 * x + 1], o[4 * x + 2], o[4 * x + 3]);
        if (grp == 0) p.ws_lse[own] = lse_own;
      }
      __threadfence();
      named_bar_sync(kBarSoftmax, 256);
      if (grp == 0 && m == 0) {
        int last = 0;
        if (*reinterpret_cast<volatile int*>(&bars->abort) == 0)
          last = (atomicAdd(&p.ws_count[unit], 1) == active - 1) ? 1 : 0;
        bars->last = last;
      }
      named_bar_sync(kBarSoftmax, 256);
      if (*reinterpret_cast<volatile int*>(&bars->last)) {
        __threadfence();
        if (ok && row_ok) {
          float M = -INFINITY, S = 0.f;
#pragma unroll
          for (int x = 0; x < 64; ++x) o[x] = 0.f;
          for (int sp = 0; sp < active; ++sp) {
            const long long slot = (unit * p.splits + sp) * kBlockM + m;
            const float ls = __ldcg(p.ws_lse + slot);
            const float4* src = reinterpret_cast<const float4*>(p.ws_o + slot * kHeadDim + col0);
            float4 v[16];
#pragma unroll
            for (int x = 0; x < 16; ++x) v[x] = __ldcg(src + x);
            const float Mn = fmaxf(M, ls);
            const float a = (M == -INFINITY) ? 0.f : fast_exp2(M - Mn);
            const float c2 = (ls == -INFINITY) ? 0.f : fast_exp2(ls - Mn);
            S = S * a + c2;
#pragma unroll
            for (int x = 0; x < 16; ++x) {
              o[4 * x + 0] = o[4 * x + 0] * a + c2 * v[x].x;
              o[4 * x + 1] = o[4 * x + 1] * a + c2 * v[x].y;
              o[4 * x + 2] = o[4 * x + 2] * a + c2 * v[x].z;
              o[4 * x + 3] = o[4 * x + 3] * a + c2 * v[x].w;
            }
            M = Mn;
          }
          store_out(o, S > 0.f ? 1.f / S : 0.f);
        }
        named_bar_sync(kBarSoftmax, 256);
        if (grp == 0 && m == 0) atomicExch(&p.ws_count[unit], 0);
      }
    }
  }

  // ---- teardown ----
  if (p.cluster && !cwaited) cluster_wait();
  // Every other split's `go` arrive has landed before this CTA's shared
  // memory goes away.
  if (cmerge && threadIdx.x == 0) wait_bar_cluster(&bars->go, 0, bars, p);
  tc_fence_before();
  __syncthreads();
  // A CTA that unwound after a failed wait may still have MMAs in flight (the
  // waits that would have seen them complete gave up): the MMA warp lets them
  // finish before the tensor memory they write is freed. The abort flag is
  // settled here (every thread has passed its last wait), so the branch is
  // uniform over the CTA.
  // Likewise the producers let their last tensor copies land (a ring that
  // finished issuing before the abort was raised has not drained), so no copy
  // writes into this CTA's shared memory after it exits.
  if (*reinterpret_cast<volatile int*>(&bars->abort) != 0) {
    if (warp == 1 && mma_issued) {
      tc_commit_elect(&bars->drain);
      mbar_wait(&bars->drain, 0, kDrainNs, nullptr);
    }
    if (warp == 0) {
      drain_ring(bars->k_full, kStagesK, issued, lane);
      if (lane == 0) mbar_wait(&bars->q_full, 0, kDrainNs, nullptr);
    } else if (warp == 2) {
      drain_ring(bars->v_full, kStagesV, issued, lane);
    }
    tc_fence_before();
    __syncthreads();
  }
  if (warp == 3) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// Paired M-tiles (paged caches). One CTA serves two M-tiles A = 2*pair and
// B = 2*pair + 1 of one (sequence, KV head) from every K/V tile it loads, so
// the tensor copies per unit of work halve; with 16-token pages the per-copy
// cost, not the tensor pipe, otherwise sets the pace.
//
// The work is a sequence of jobs, one per (tile, M-tile): with B present,
// job j is M-tile j & 1 of tile j >> 1; without B (a sequence too short for
// it), job j is tile j of A. Job j's S goes to TMEM columns [128 (j & 1), +128)
// (S_A / S_B, or S double-buffered for A alone); each M-tile has one O
// accumulator, O_A [256, 384) and O_B [384, 512). The MMA order is the single
// M-tile kernel's with jobs for tiles: Q*K^T(0), Q*K^T(1), then P*V(j),
// Q*K^T(j + 2); one thread's MMAs complete in order, so Q*K^T(j + 2) cannot
// overwrite P(j) before P*V(j) has read it, and a completed Q*K^T(j) implies
// P*V(j - 2) has completed.
//
// Both softmax groups work on every job: group g takes keys [64g, 64g + 64)
// of the tile, but the two share the row maximum (each leaves its half's
// maximum in a shared-memory buffer of the job's parity, the quadrant's two
// warps meet at a named barrier, and each reads the other's), so one O per M-tile
// suffices: each group rescales and finishes columns [64g, 64g + 64) of it,
// and the groups' row sums add at the end. The key range is not split (one
// CTA per pair).
constexpr int kPairStagesK = 2;
constexpr int kPairStagesV = 2;
constexpr uint32_t kPOffQ = 0;                                   // Q_A, then Q_B
constexpr uint32_t kPOffK = 2 * kTileBytes;
constexpr uint32_t kPOffV = kPOffK + kPairStagesK * kTileBytes;
// The row maxima the two softmax warps of a row trade each job,
// [job parity][group][row]: one buffer per parity, so a warp's write for job
// j + 2 comes after barrier j + 1, which the other warp reaches only once it
// has read job j's value.
constexpr uint32_t kPOffX = kPOffV + kPairStagesV * kTileBytes;
constexpr uint32_t kPOffBar = kPOffX + 2 * 2 * 128 * sizeof(float);

struct PairBars {
  uint64_t q_full;
  uint64_t k_full[kPairStagesK];
  uint64_t k_empty[kPairStagesK];
  uint64_t v_full[kPairStagesV];
  uint64_t v_empty[kPairStagesV];
  uint64_t s_full[2];   // [j & 1]: Q*K^T(j) has completed (phase j >> 1)
  uint64_t p_full[2];   // [j & 1]: P(j) is written (8 warps, phase j >> 1)
  uint64_t o_done[2];   // [j & 1]: P*V(j) has completed (phase j >> 1)
  uint64_t drain;
  uint64_t staged;
  uint64_t stage_issued;
  uint64_t stall;
  uint32_t tmem_base;
  int abort;
};

constexpr uint32_t kPairSmemBytes = kPOffBar + ((sizeof(PairBars) + 127) / 128) * 128 + 1024;
static_assert(kPairSmemBytes <= 232448, "shared memory budget (paired M-tiles)");

__global__ void __launch_bounds__(kThreads, 1)
slot_attn_pair_kernel(const __grid_constant__ CUtensorMap map_q,
                      const __grid_constant__ CUtensorMap map_k,
                      const __grid_constant__ CUtensorMap map_v, const TcParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  PairBars* bars = reinterpret_cast<PairBars*>(smem + kPOffBar);
  float* xmax = reinterpret_cast<float*>(smem + kPOffX);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  // the work tile, from the grid or the schedule (read after the wait)
  const int pos = blockIdx.z * gridDim.x + blockIdx.x;
  int pair = blockIdx.x;
  int b = blockIdx.z / p.Hkv;
  int kvh = blockIdx.z - b * p.Hkv;
  bool sched_ok = true;

  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&map_q);
    tma_prefetch_map(&map_k);
    tma_prefetch_map(&map_v);
  }
  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    for (int s = 0; s < kPairStagesK; ++s) {
      mbar_init(&bars->k_full[s], 1);
      mbar_init(&bars->k_empty[s], 1);
    }
    for (int s = 0; s < kPairStagesV; ++s) {
      mbar_init(&bars->v_full[s], 1);
      mbar_init(&bars->v_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&bars->s_full[s], 1);
      mbar_init(&bars->p_full[s], kSoftmaxWarps);
      mbar_init(&bars->o_done[s], 1);
    }
    mbar_init(&bars->drain, 1);
    mbar_init(&bars->staged, kSoftmaxWarps);
    mbar_init(&bars->stage_issued, kSoftmaxWarps);
    mbar_init(&bars->stall, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  // every barrier is initialised before any thread touches one
  __syncthreads();
  // warp 1 holds the tensor memory, warp 3 issues the MMAs (its SM
  // sub-partition's softmax warps measured least slowed by the issuer)
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 || warp == 2) named_bar_arrive(kBarSetup, kThreads);
  // Inputs may be written by the kernel launched before this one.
  grid_dependency_wait();
  if (p.perm != nullptr) sched_ok = scheduled_tile(p, p.perm[pos / p.Hkv], pos, b, kvh, pair);
  if (!sched_ok) b = 0;   // reported below; no work is done

  // ---- per-sequence geometry (uniform over the CTA) ----
  const int P = p.cache_lens[b];
  const long long R64 = static_cast<long long>(p.n_slots[b]) * p.slot_len[b];
  const int R = R64 > p.max_rows ? p.max_rows + 1 : static_cast<int>(R64);
  const int mode = p.mask_mode[b];
  const int row0 = p.q_row_offsets[b];
  const int row_end = p.q_row_offsets[b + 1];
  int code = 0;
  if (!sched_ok)
    code = ZARYA_DEVERR_ROWS;
  else if (mode != ZARYA_MASK_BIDIR_BLOCK && mode != ZARYA_MASK_SLOT_CAUSAL &&
           mode != ZARYA_MASK_SLOT_INDEPENDENT)
    code = ZARYA_DEVERR_MASK_MODE;
  else if (p.n_slots[b] < 1 || p.slot_len[b] < 1 || R > p.max_rows || row_end - row0 != R ||
           row0 < 0 || row_end > p.total_rows)
    code = ZARYA_DEVERR_ROWS;
  else if (P < 0 || static_cast<long long>(P) + R > p.capacity) code = ZARYA_DEVERR_CAPACITY;
  const int rows_per_tile = kBlockM / p.g;
  const int r0A = 2 * pair * rows_per_tile;
  const int r0B = r0A + rows_per_tile;
  const bool hasB = r0B < R;
  const int r_hi = min(r0A + 2 * rows_per_tile, R) - 1;   // last block row of the pair
  const int kv_end = (mode == ZARYA_MASK_BIDIR_BLOCK) ? P + R : P + r_hi + 1;
  const int nt = (code != 0 || kv_end <= 0) ? 1 : (kv_end + kBlockN - 1) / kBlockN;
  const int njobs = hasB ? 2 * nt : nt;
  const int jshift = hasB ? 1 : 0;   // tile of job j = j >> jshift
  int st_lo = 0, st_hi = 0;   // staged attention: block rows read, relative to P
  if (p.k_new != nullptr && code == 0) st_hi = kv_end - P;

  const bool works = code == 0 && r0A < R;
  const int t_stage = st_hi > st_lo ? P / kBlockN : -1;
  int issued = 0;
  const bool stage_here = works && st_hi > st_lo;
  GroupStager stg;
  if (warp >= 4 && stage_here) {
    stg.load(p, b, kvh, row0, P, st_lo, st_hi, threadIdx.x - 128, 0);
    __syncwarp();
    if (lane == 0) mbar_arrive_relaxed(&bars->stage_issued);
  }
  if (warp == 0 && works && lane == 0) {
    // Q of both M-tiles (B's rows past R_b are never stored)
    mbar_arrive_expect_tx(&bars->q_full, (hasB ? 2u : 1u) * kTileBytes);
    const uint32_t dq = smem_u32(smem + kPOffQ);
    tma_load_3d(dq, &map_q, &bars->q_full, 0, kvh * p.g, row0 + r0A);
    tma_load_3d(dq + kHalfBytes, &map_q, &bars->q_full, 64, kvh * p.g, row0 + r0A);
    if (hasB) {
      tma_load_3d(dq + kTileBytes, &map_q, &bars->q_full, 0, kvh * p.g, row0 + r0B);
      tma_load_3d(dq + kTileBytes + kHalfBytes, &map_q, &bars->q_full, 64, kvh * p.g, row0 + r0B);
    }
  }
  if ((warp == 0 || warp == 2) && works && stage_here) {
    // a timeout sets the abort flag; the ring loop below then returns early
    if (lane == 0) wait_bar(&bars->stage_issued, 0, bars, p);
    __syncwarp();
  }
  if (warp != 0 && warp != 2) {
    tc_fence_before();
    named_bar_sync(kBarSetup, kThreads);
    tc_fence_after();
  }
  const uint32_t tmem = (warp != 0 && warp != 2) ? bars->tmem_base : 0u;
  bool mma_issued = false;
  if (!works) {
    if (code != 0 && (pair == 0 || !sched_ok) && threadIdx.x == 0) record_error(p.err, code);
    grid_launch_dependents();
    if (warp == 1) tmem_dealloc(tmem, kTmemCols);
    return;
  }

  if (warp < 4) {
    if (warp == 0) {
      if (!produce_range(&map_k, bars->k_full, bars->k_empty, kPairStagesK,
                         smem_u32(smem + kPOffK), p, bars, b, kvh, 0, 0, nt, kv_end, lane, t_stage,
                         issued))
        drain_ring(bars->k_full, kPairStagesK, issued, lane);
      if (lane == 0 && *reinterpret_cast<volatile int*>(&bars->abort) != 0)
        mbar_wait(&bars->q_full, 0, kDrainNs, nullptr);
    } else if (warp == 2) {
      if (!produce_range(&map_v, bars->v_full, bars->v_empty, kPairStagesV,
                         smem_u32(smem + kPOffV), p, bars, b, kvh, 0, 0, nt, kv_end, lane, t_stage,
                         issued))
        drain_ring(bars->v_full, kPairStagesV, issued, lane);
    } else if (warp == 3) {
      // ======================= MMA issuer (one elected lane) =======================
      bool ok = true;
      if (p.debug_stall) ok = wait_bar(&bars->stall, 0, bars, p);
      if (ok) ok = wait_bar(&bars->q_full, 0, bars, p);
      bool any_mma = false;
      tc_fence_after();
      const uint32_t q0 = smem_u32(smem + kPOffQ);
      const uint64_t k_desc0 = sdesc_sw128(smem_u32(smem + kPOffK), 16, 1024);
      const uint64_t v_desc0 = sdesc_sw128(smem_u32(smem + kPOffV), kHalfBytes, 1024);
      constexpr uint64_t kTileUnits = kTileBytes >> 4, kHalfUnits = kHalfBytes >> 4;
      // A tile's first job waits for its K (V) tile; its last job releases it.
      auto first_of_tile = [&](int j) { return !hasB || (j & 1) == 0; };
      auto last_of_tile = [&](int j) { return !hasB || (j & 1) == 1; };
      auto issue_qk = [&](int j) -> bool {
        const int i = j >> jshift;
        const int s = i % kPairStagesK;
        const int t = hasB ? (j & 1) : 0;
        if (first_of_tile(j)) {
          if (!wait_bar(&bars->k_full[s], (i / kPairStagesK) & 1, bars, p)) return false;
          tc_fence_after();
        }
        const uint32_t qt = q0 + t * kTileBytes;
        const uint64_t qd0 = sdesc_sw128(qt, 16, 1024);
        const uint64_t qd1 = sdesc_sw128(qt + kHalfBytes, 16, 1024);
        const uint64_t kd = k_desc0 + s * kTileUnits;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t step = (kk >> 2) * kHalfUnits + (kk & 3) * 2;
          tc_mma_ss_elect(tmem + (j & 1) * 128, (kk < 4 ? qd0 : qd1) + (kk & 3) * 2, kd + step,
                          kIdescQK, kk > 0 ? 1u : 0u);
        }
        any_mma = true;
        tc_commit_elect(&bars->s_full[j & 1]);
        if (last_of_tile(j)) tc_commit_elect(&bars->k_empty[s]);
        return true;
      };
      // O_t += P(j) V: group g's P is packed over columns [64g, 64g + 32) of S(j)
      auto issue_pv = [&](int j) -> bool {
        const int i = j >> jshift;
        const int sv = i % kPairStagesV;
        const int t = hasB ? (j & 1) : 0;
        if (!wait_bar(&bars->p_full[j & 1], (j >> 1) & 1, bars, p)) return false;
        if (first_of_tile(j)) {
          if (!wait_bar(&bars->v_full[sv], (i / kPairStagesV) & 1, bars, p)) return false;
        }
        tc_fence_after();
        const uint64_t vd = v_desc0 + sv * kTileUnits;
#pragma unroll
        for (int c = 0; c < 8; ++c)
          tc_mma_ts_elect(tmem + kTmemO + t * 128, tmem + (j & 1) * 128 + (c >> 2) * 64 + (c & 3) * 8,
                          vd + c * 128, kIdescPV, (i > 0 || c > 0) ? 1u : 0u);
        any_mma = true;
        tc_commit_elect(&bars->o_done[j & 1]);
        if (last_of_tile(j)) tc_commit_elect(&bars->v_empty[sv]);
        return true;
      };
      if (ok) ok = issue_qk(0);
      if (ok && njobs > 1) ok = issue_qk(1);
      for (int j = 0; j < njobs && ok; ++j) {
        if (!issue_pv(j)) { ok = false; break; }
        if (j + 2 < njobs && !issue_qk(j + 2)) { ok = false; break; }
      }
      mma_issued = any_mma;
    }
  } else {
    // ======================= softmax + epilogue =======================
    if (stage_here) {
      stg.finish(p, b, kvh, row0, P, st_lo, st_hi, threadIdx.x - 128);
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->staged);
    }
    const int grp = (warp - 4) >> 2;
    const int wq = warp & 3;
    const int m = wq * 32 + lane;   // packed row = TMEM lane (of both M-tiles)
    const int h = kvh * p.g + (m - (m / p.g) * p.g);
    // this lane's block row of M-tile t is r0A + t * rows_per_tile + mrow
    const int mrow = m / p.g;
    const int L = p.slot_len[b];
    auto row_of = [&](int t) { return r0A + t * rows_per_tile + mrow; };
    auto row_valid = [&](int t) { return row_of(t) < R && (t == 0 || hasB); };
    const uint32_t t_row = tmem + (static_cast<uint32_t>(wq * 32) << 16);
    const float sl2 = p.scale_log2;
    float m_runA = -INFINITY, m_runB = -INFINITY;
    float l_runA = 0.f, l_runB = 0.f;
    bool ok = true;
    auto mask64 = [&](float (&s)[64], int c0, int limit, int hide_hi) {
      if (c0 + 64 > limit) {
#pragma unroll
        for (int x = 0; x < 64; ++x)
          if (c0 + x >= limit) s[x] = -INFINITY;
      }
      if (hide_hi > P && c0 < hide_hi && c0 + 64 > P) {
#pragma unroll
        for (int x = 0; x < 64; ++x)
          if (c0 + x >= P && c0 + x < hide_hi) s[x] = -INFINITY;
      }
    };
    for (int j = 0; j < njobs; ++j) {
      const int i = j >> jshift;
      const int t = hasB ? (j & 1) : 0;
      const int rt = row_of(t);
      const bool okt = row_valid(t);
      const int limit = !okt ? kv_end : (mode == ZARYA_MASK_BIDIR_BLOCK ? P + R : P + rt + 1);
      const int hide_hi = (okt && mode == ZARYA_MASK_SLOT_INDEPENDENT) ? P + (rt / L) * L : P;
      const uint32_t t_s = t_row + (j & 1) * 128;
      const uint32_t t_o = t_row + kTmemO + t * 128 + grp * 64;
      const int c_tile = i * kBlockN;
      const int c0 = c_tile + grp * 64;   // this group's keys
      if (ok) ok = wait_bar(&bars->s_full[j & 1], (j >> 1) & 1, bars, p);
      ok = __all_sync(0xffffffffu, ok);
      // This group's scores and their row maximum, which it leaves in shared
      // memory for the other group of the row.
      float s[64];
      float mx = -INFINITY;
      if (ok) {
        tc_fence_after();
        tmem_ld_32x32b_x64(t_s + grp * 64, s);
        mask64(s, c0, limit, hide_hi);
        mx = max64(s);
        xmax[((j & 1) * 2 + grp) * 128 + m] = mx;
      }
      // Both warps of the quadrant arrive here every job and leave together,
      // going on only if both got their S; the barrier orders their shared-
      // memory writes before the reads, and each reads the other's maximum.
      if (!named_bar_and(2 + wq, 64, ok)) { ok = false; break; }
      mx = fmaxf(mx, xmax[((j & 1) * 2 + (1 - grp)) * 128 + m]);
      float m_run = t ? m_runB : m_runA;
      float l_run = t ? l_runB : l_runA;
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
      // Rescaling this group's half of O_t must wait for the last P*V that
      // wrote O_t: job j - 2 with B present, j - 1 without (the S of job j
      // completing implies P*V(j - 2) has completed, so neither parity wait
      // can alias an older phase).
      if (warp_need && i > 0) {
        const int jp = hasB ? j - 2 : j - 1;
        if (ok) ok = wait_bar(&bars->o_done[jp & 1], (jp >> 1) & 1, bars, p);
        tc_fence_after();
#pragma unroll
        for (int ch = 0; ch < 2; ++ch) {
          float v[32];
          const uint32_t a = t_o + ch * 32;
          tmem_ld_32x32b_x32(a, v);
#pragma unroll
          for (int x = 0; x < 32; ++x) v[x] *= alpha;
          tmem_st_32x32b_x32(a, v);
        }
      }
      // Keys at or past kv_end in the last tile: their V rows must be exact
      // zeros before the tile's first P*V reads them; each group clears the
      // rows of its half.
      if ((!hasB || t == 0) && c0 + 64 > kv_end) {
        const int sv = i % kPairStagesV;
        if (ok) ok = wait_bar(&bars->v_full[sv], (i / kPairStagesV) & 1, bars, p);
        const int key = grp * 64 + (m & 63);
        if (ok && m < 64 && c0 + (m & 63) >= kv_end) {
          uint8_t* vrow = smem + kPOffV + sv * kTileBytes + (key >> 3) * 1024 + (key & 7) * 128;
          const uint4 z = make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
          for (int x = 0; x < 8; ++x) {
            reinterpret_cast<uint4*>(vrow)[x] = z;
            reinterpret_cast<uint4*>(vrow + kHalfBytes)[x] = z;
          }
        }
        fence_proxy_async_smem();
      }
      // P = 2^(s * scale * log2 e - m) for this group's keys, packed bf16
      // pairs over the first 32 columns of its half of S.
      float pk[32];
      l_run += exp_pack_row(s, sl2, m_use, pk);
      tmem_st_32x32b_x32(t_s + grp * 64, pk);
      if (t) {
        m_runB = m_run;
        l_runB = l_run;
      } else {
        m_runA = m_run;
        l_runA = l_run;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->p_full[j & 1]);
    }

    // ---- epilogue: the groups' row sums add (both used the same maxima);
    // the Q buffer (read by no MMA any more) carries them ----
    float* xch = reinterpret_cast<float*>(smem + kPOffQ);
    xch[(grp * 2 + 0) * 128 + m] = l_runA;
    xch[(grp * 2 + 1) * 128 + m] = l_runB;
    named_bar_sync(kBarSoftmax, 256);
    const float l_totA = xch[m] + xch[2 * 128 + m];
    const float l_totB = xch[128 + m] + xch[3 * 128 + m];
    grid_launch_dependents();
    // P*V(njobs - 1) completes after every other MMA of the CTA
    if (ok) ok = wait_bar(&bars->o_done[(njobs - 1) & 1], ((njobs - 1) >> 1) & 1, bars, p);
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();
#pragma unroll
    for (int t = 0; t < 2; ++t) {
      if (ok && row_valid(t)) {
        const float l_tot = t ? l_totB : l_totA;
        const float inv = (l_tot > 0.f) ? 1.f / l_tot : 0.f;
        float o[64];
        tmem_ld_32x32b_x64(t_row + kTmemO + t * 128 + grp * 64, o);
        uint4* d4 = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(p.out) +
                                             (static_cast<long long>(row0 + row_of(t)) * p.Hq +
                                              h) * kHeadDim + grp * 64);
#pragma unroll
        for (int x = 0; x < 8; ++x)
          d4[x] = make_uint4(pack_bf16(o[8 * x + 0] * inv, o[8 * x + 1] * inv),
                             pack_bf16(o[8 * x + 2] * inv, o[8 * x + 3] * inv),
                             pack_bf16(o[8 * x + 4] * inv, o[8 * x + 5] * inv),
                             pack_bf16(o[8 * x + 6] * inv, o[8 * x + 7] * inv));
      }
    }
  }

  // ---- teardown (as the single-tile kernel's) ----
  tc_fence_before();
  __syncthreads();
  if (*reinterpret_cast<volatile int*>(&bars->abort) != 0) {
    if (warp == 3 && mma_issued) {
      tc_commit_elect(&bars->drain);
      mbar_wait(&bars->drain, 0, kDrainNs, nullptr);
    }
    if (warp == 0) {
      drain_ring(bars->k_full, kPairStagesK, issued, lane);
      if (lane == 0) mbar_wait(&bars->q_full, 0, kDrainNs, nullptr);
    } else if (warp == 2) {
      drain_ring(bars->v_full, kPairStagesV, issued, lane);
    }
    tc_fence_before();
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// Dispatch order. A launch of several waves runs its CTAs in grid order as SMs
// free up, so a long work tile dispatched late sets the end of the launch
// (serving_mix: SMs busy 85 % of the launch). For paired launches of several
// waves this one-CTA kernel sorts the work items (sequence, M-tile or pair) by cost
// (M-tiles x key tiles: the tile loop's work), largest first, ties in item
// order, and the attention CTA at position pos serves item perm[pos / Hkv],
// KV head pos % Hkv: the greedy longest-first order. Items a CTA would find
// empty (or invalid: the attention kernel reports those) cost 0 and go last.
constexpr int kSchedThreads = 1024;

__global__ void __launch_bounds__(kSchedThreads) schedule_kernel(const TcParams p) {
  __shared__ unsigned long long key[kMaxSchedItems];
  grid_dependency_wait();
  const int T = p.items;
  const int N = p.B * T;
  int n2 = 1;
  while (n2 < N) n2 <<= 1;
  const int rows_per_tile = kBlockM / p.g;
  const int span = p.pair ? 2 : 1;   // M-tiles per item
  for (int i = threadIdx.x; i < n2; i += kSchedThreads) {
    unsigned long long k = ~0ull;
    if (i < N) {
      const int b = i / T, t = i - b * T;
      const int P = p.cache_lens[b];
      const long long R64 = static_cast<long long>(p.n_slots[b]) * p.slot_len[b];
      const int mode = p.mask_mode[b];
      uint32_t cost = 0;
      if (P >= 0 && R64 >= 1 && R64 <= p.max_rows && P + R64 <= p.capacity) {
        const int R = static_cast<int>(R64);
        const int r0 = span * t * rows_per_tile;
        if (r0 < R) {
          const int m = min(span, (R - r0 + rows_per_tile - 1) / rows_per_tile);
          const int r_hi = min(r0 + span * rows_per_tile, R) - 1;
          const int kv_end = mode == ZARYA_MASK_BIDIR_BLOCK ? P + R : P + r_hi + 1;
          cost = static_cast<uint32_t>(m) * static_cast<uint32_t>((kv_end + kBlockN - 1) / kBlockN) + 1;
        }
      }
      k = (static_cast<unsigned long long>(0xFFFFFFFFu - cost) << 32) | static_cast<uint32_t>(i);
    }
    key[i] = k;
  }
  __syncthreads();
  // bitonic sort, ascending key = descending cost
  for (int size = 2; size <= n2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = threadIdx.x; i < n2; i += kSchedThreads) {
        const int j = i ^ stride;
        if (j > i) {
          const bool up = (i & size) == 0;
          const unsigned long long a = key[i], c = key[j];
          if ((a > c) == up) {
            key[i] = c;
            key[j] = a;
          }
        }
      }
      __syncthreads();
    }
  }
  int32_t* perm = const_cast<int32_t*>(p.perm);
  for (int k = threadIdx.x; k < N; k += kSchedThreads)
    perm[k] = static_cast<int32_t>(key[k] & 0xFFFFFFFFull);
  grid_launch_dependents();
}

}  // namespace

size_t tc_smem_bytes() { return kSmemBytes; }

cudaError_t launch_schedule(const TcParams& p, cudaStream_t stream) {
  PdlLaunch l(dim3(1), dim3(kSchedThreads), 0, stream);
  return cudaLaunchKernelEx(&l.cfg, schedule_kernel, p);
}

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
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(slot_attn_pair_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(kPairSmemBytes));
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  cudaLaunchConfig_t cfg{};
  cudaLaunchAttribute attr[2]{};
  cfg.gridDim = dim3(p.pair ? (p.m_tiles + 1) / 2 : p.m_tiles, p.splits, p.B * p.Hkv);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = p.pair ? kPairSmemBytes : kSmemBytes;
  cfg.stream = stream;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.numAttrs = 1;
  if (p.cluster) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 1;
    attr[1].val.clusterDim.y = p.splits;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
  }
  cfg.attrs = attr;
  if (p.pair) return cudaLaunchKernelEx(&cfg, slot_attn_pair_kernel, map_q, map_k, map_v, p);
  return cudaLaunchKernelEx(&cfg, slot_attn_tc_kernel, map_q, map_k, map_v, p);
}

}  // namespace zarya
