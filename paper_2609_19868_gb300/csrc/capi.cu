// Host side of the C ABI declared in include/zarya.h: argument validation,
// device selection, TMA tensor-map encoding, split planning, workspace
// layout and kernel launches. Allocates nothing.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <cstdio>

#include "internal.cuh"
#include "token_ops.cuh"

namespace zarya {
namespace {

constexpr int32_t kVersion = 200;  // 0.2.0

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int sm_count() {
  constexpr int kMaxDevices = 64;
  static int cache[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 148;
  int n = __atomic_load_n(&cache[dev], __ATOMIC_ACQUIRE);
  if (n == 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
      n = 148;
    __atomic_store_n(&cache[dev], n, __ATOMIC_RELEASE);
  }
  return n;
}

zarya_status check_desc(const zarya_attn_desc* d) {
  if (d == nullptr) return ZARYA_ERR_INVALID_ARG;
  if (d->batch < 1 || d->n_q_heads < 1 || d->n_kv_heads < 1 || d->head_dim < 1)
    return ZARYA_ERR_INVALID_ARG;
  if (d->n_q_heads % d->n_kv_heads != 0) return ZARYA_ERR_INVALID_ARG;
  if (d->dtype != ZARYA_BF16 && d->dtype != ZARYA_FP32) return ZARYA_ERR_INVALID_ARG;
  if (d->page_size < 0 || d->cache_capacity < 1 || d->max_rows < 1 || d->total_rows < 1 ||
      d->max_kv_len < 0 || d->kv_splits < 0 || d->n_pages < 0)
    return ZARYA_ERR_INVALID_ARG;
  if (!(d->scale >= 0.f) || std::isinf(d->scale)) return ZARYA_ERR_INVALID_ARG;
  if (d->q_row_offsets == nullptr) return ZARYA_ERR_INVALID_ARG;
  if (d->wait_limit_us < 0 || (d->debug_flags & ~ZARYA_DEBUG_STALL) != 0)
    return ZARYA_ERR_INVALID_ARG;
  if (d->page_size > 0) {
    if (d->cache_capacity % d->page_size != 0 || d->n_pages < 1) return ZARYA_ERR_INVALID_ARG;
  }
  if (static_cast<long long>(d->batch) * d->cache_capacity > 0x7fffffffLL &&
      d->page_size == 0)
    return ZARYA_ERR_UNSUPPORTED;
  const int eb = d->dtype == ZARYA_BF16 ? 2 : 4;
  if ((static_cast<long long>(d->n_kv_heads) * d->head_dim * eb) % 16 != 0)
    return ZARYA_ERR_UNSUPPORTED;
  return ZARYA_OK;
}

// Attention-specific support checks.
zarya_status check_attn_support(const zarya_attn_desc* d) {
  if (d->dtype == ZARYA_BF16) {
    if (d->head_dim != kHeadDim) return ZARYA_ERR_UNSUPPORTED;
    const int g = d->n_q_heads / d->n_kv_heads;
    if (g > kBlockM || kBlockM % g != 0) return ZARYA_ERR_UNSUPPORTED;
    if (d->page_size != 0 && d->page_size != 16 && d->page_size != 32 && d->page_size != 64 &&
        d->page_size != 128)
      return ZARYA_ERR_UNSUPPORTED;
  } else {
    if (d->head_dim % 32 != 0 || d->head_dim > 256) return ZARYA_ERR_UNSUPPORTED;
  }
  return ZARYA_OK;
}


struct Plan {
  int g, m_tiles, splits;
  int pair;   // one CTA per pair of M-tiles (grid.x = pairs)
  int items;  // work items per sequence: M-tiles, or pairs of them
  int sched;  // longest-first dispatch order, in the workspace at offset 0
  size_t cnt_bytes;   // split arrival counters at the end of the workspace
  long long units;
  size_t off_lse, off_cnt, bytes;
};

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// A paired launch of several waves gets a dispatch order: its work items
// sorted longest first by a one-CTA kernel into the workspace (B x items
// int32), which the attention CTAs follow (a long tile dispatched late would
// otherwise set the end of the launch: serving_mix 772 -> 726 us). Measured
// and not taken for the single-tile kernel: ragged_mid ran 2-3 % slower with
// it (the order did not shorten its tail, and the mapping cost the tile loop).
Plan with_schedule(Plan p, const zarya_attn_desc* d, int sms) {
  p.items = p.pair ? (p.m_tiles + 1) / 2 : p.m_tiles;
  const long long items = static_cast<long long>(d->batch) * p.items;
  if (p.pair && items * d->n_kv_heads > sms && items <= kMaxSchedItems) {
    p.sched = 1;
    p.bytes = align256(static_cast<size_t>(items) * sizeof(int32_t));
  }
  return p;
}

// Split-KV plan of the tensor-core path: the key range of every work tile
// (sequence, KV head, M-tile) is split so that the slowest SM (waves x tiles
// per CTA, plus a fixed per-CTA cost) is as short as possible. Splitting also
// pays when the tiles already fill the GPU but leave a partial last wave
// (long_ctx: 512 tiles are 3.4 waves of 152 SMs; two splits make 6.7).
Plan plan_tc(const zarya_attn_desc* d, int sms) {
  Plan p{};
  p.g = d->n_q_heads / d->n_kv_heads;
  p.m_tiles = static_cast<int>((static_cast<long long>(d->max_rows) * p.g + kBlockM - 1) / kBlockM);
  p.units = static_cast<long long>(d->batch) * d->n_kv_heads * p.m_tiles;
  const long long kv_max = d->max_kv_len > 0 ? d->max_kv_len : d->cache_capacity;
  const int tiles = static_cast<int>((kv_max + kBlockN - 1) / kBlockN);
  // Paged caches cost one tensor copy per page per tile; serving two M-tiles
  // of a (sequence, KV head) from each tile halves the copies per unit of
  // work. Taken when the pairs alone fill the GPU (no key split needed).
  const long long pairs = (p.m_tiles + 1) / 2;
  if (d->page_size > 0 && d->kv_splits == 0 && p.m_tiles >= 2 &&
      static_cast<long long>(d->batch) * d->n_kv_heads * pairs >= sms) {
    p.pair = 1;
    p.splits = 1;
    return with_schedule(p, d, sms);
  }
  int splits = 1;
  if (d->kv_splits > 0) {
    splits = d->kv_splits < tiles ? d->kv_splits : tiles;
  } else {
    double best = 1e30;
    for (int s = 1; s <= tiles && s <= kMaxClusterSplits; ++s) {
      const long long waves = (p.units * s + sms - 1) / sms;
      const double cost = static_cast<double>(waves) * ((tiles + s - 1) / s + 2.0) +
                          (s > 1 ? 1.0 : 0.0);
      if (cost < best - 1e-9) {
        best = cost;
        splits = s;
      }
    }
  }
  if (splits < 1) splits = 1;
  p.splits = splits;
  // Up to kMaxClusterSplits splits merge through distributed shared memory
  // inside a thread-block cluster; more splits merge through the workspace.
  if (splits > kMaxClusterSplits) {
    const size_t n = static_cast<size_t>(p.units) * splits * kBlockM;
    const size_t bytes_o = n * kHeadDim * sizeof(float);
    p.off_lse = align256(bytes_o);
    p.off_cnt = align256(p.off_lse + n * sizeof(float));
    p.bytes = align256(p.off_cnt + static_cast<size_t>(p.units) * sizeof(int32_t));
    p.cnt_bytes = p.bytes - p.off_cnt;
  }
  return with_schedule(p, d, sms);
}

CUresult encode(CUtensorMap* map, void* base, cuuint32_t rank, const cuuint64_t* dims,
                const cuuint64_t* strides, const cuuint32_t* box) {
  auto fn = tensor_map_encoder();
  if (fn == nullptr) return CUDA_ERROR_NOT_FOUND;
  const cuuint32_t es[4] = {1, 1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, base, dims, strides, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

}  // namespace

// Makes the device that owns `stream` current for this thread. The stream is
// asked directly unless it is capturing into a CUDA graph (where that query is
// not permitted) or is the legacy default stream; then the device that owns
// `ptr` (a device buffer of the call) is used.
cudaError_t select_device(cudaStream_t stream, const void* ptr) {
  int want = -1;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (stream != nullptr) {
    cudaError_t e = cudaStreamIsCapturing(stream, &cs);
    if (e != cudaSuccess) return e;
  }
  if (stream != nullptr && cs == cudaStreamCaptureStatusNone) {
    cudaError_t e = cudaStreamGetDevice(stream, &want);
    if (e != cudaSuccess) return e;
  } else {
    cudaPointerAttributes attr{};
    cudaError_t e = cudaPointerGetAttributes(&attr, ptr);
    if (e != cudaSuccess) return e;
    if (attr.type != cudaMemoryTypeDevice && attr.type != cudaMemoryTypeManaged)
      return cudaErrorInvalidValue;
    want = attr.device;
  }
  int cur = -1;
  cudaError_t e = cudaGetDevice(&cur);
  if (e != cudaSuccess) return e;
  if (cur != want) return cudaSetDevice(want);
  return cudaSuccess;
}

static thread_local char g_last_error[256] = "";

zarya_status cuda_fail(const char* what, cudaError_t e) {
  std::snprintf(g_last_error, sizeof g_last_error, "%s: %s (%d)", what, cudaGetErrorString(e),
                static_cast<int>(e));
  return ZARYA_ERR_CUDA;
}

size_t workspace_counter_bytes(const zarya_attn_desc* desc) {
  if (check_desc(desc) != ZARYA_OK || check_attn_support(desc) != ZARYA_OK) return 0;
  if (desc->dtype != ZARYA_BF16) return 0;
  return plan_tc(desc, sm_count()).cnt_bytes;
}

}  // namespace zarya

using namespace zarya;

extern "C" {

const char* zarya_slot_attn_kernel(const zarya_attn_desc* desc) {
  if (check_desc(desc) != ZARYA_OK || check_attn_support(desc) != ZARYA_OK) return "none";
  if (desc->dtype != ZARYA_BF16) return "slot_attn_f32_kernel";
  return plan_tc(desc, sm_count()).pair ? "slot_attn_pair_kernel" : "slot_attn_tc_kernel";
}

int32_t zarya_slot_attn_launches(const zarya_attn_desc* desc) {
  if (check_desc(desc) != ZARYA_OK || check_attn_support(desc) != ZARYA_OK) return 0;
  if (desc->dtype != ZARYA_BF16) return 1;
  return plan_tc(desc, sm_count()).sched ? 2 : 1;
}

size_t zarya_slot_attn_workspace_size(const zarya_attn_desc* desc) {
  if (check_desc(desc) != ZARYA_OK || check_attn_support(desc) != ZARYA_OK) return 0;
  if (desc->dtype != ZARYA_BF16) return 0;
  return plan_tc(desc, sm_count()).bytes;
}

namespace {

zarya_status kv_append_impl(const void* k_new, const void* v_new, const int32_t* accept_len,
                            void* k_cache, void* v_cache, const int32_t* cache_lens,
                            int32_t* new_lens, const int32_t* page_table, bool commit,
                            const zarya_attn_desc* desc, zarya_stream_t stream_);

// Attention, optionally staging the block's own K/V (k_new / v_new) first.
zarya_status slot_attn_impl(const void* q, const void* k_new, const void* v_new,
                            const void* k_cache, const void* v_cache, const int32_t* cache_lens,
                            const int32_t* page_table, const int32_t* n_slots,
                            const int32_t* slot_len, const int32_t* mask_mode, void* out,
                            void* workspace, size_t workspace_bytes, const zarya_attn_desc* desc,
                            zarya_stream_t stream_) {
  zarya_status st = check_desc(desc);
  if (st != ZARYA_OK) return st;
  st = check_attn_support(desc);
  if (st != ZARYA_OK) return st;
  if (!q || !k_cache || !v_cache || !cache_lens || !n_slots || !slot_len || !mask_mode || !out)
    return ZARYA_ERR_INVALID_ARG;
  const bool staged = k_new != nullptr || v_new != nullptr;
  if (staged && (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new)))
    return ZARYA_ERR_INVALID_ARG;
  if ((desc->page_size > 0) != (page_table != nullptr)) return ZARYA_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(out))
    return ZARYA_ERR_INVALID_ARG;
  if (staged && desc->dtype == ZARYA_FP32) {
    // The CUDA-core path stages with the append kernel, then attends.
    st = kv_append_impl(k_new, v_new, nullptr, const_cast<void*>(k_cache),
                        const_cast<void*>(v_cache), cache_lens, nullptr, page_table, false, desc,
                        stream_);
    if (st != ZARYA_OK) return st;
  }
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, q);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  const float scale =
      desc->scale > 0.f ? desc->scale : 1.0f / std::sqrt(static_cast<float>(desc->head_dim));
  const int max_pages = desc->page_size > 0 ? desc->cache_capacity / desc->page_size : 0;

  if (desc->dtype == ZARYA_FP32) {
    SimtParams p{};
    p.q = q;
    p.k_cache = k_cache;
    p.v_cache = v_cache;
    p.cache_lens = cache_lens;
    p.page_table = page_table;
    p.n_slots = n_slots;
    p.slot_len = slot_len;
    p.mask_mode = mask_mode;
    p.q_row_offsets = desc->q_row_offsets;
    p.out = out;
    p.err = err;
    p.B = desc->batch;
    p.Hq = desc->n_q_heads;
    p.Hkv = desc->n_kv_heads;
    p.D = desc->head_dim;
    p.max_rows = desc->max_rows;
    p.total_rows = desc->total_rows;
    p.capacity = desc->cache_capacity;
    p.page_size = desc->page_size;
    p.max_pages = max_pages;
    p.n_pages = desc->n_pages;
    p.scale = scale;
    ce = launch_slot_attn_f32(p, stream);
    return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching slot_attn_f32_kernel", ce);
  }

  const Plan plan = plan_tc(desc, sm_count());
  if (plan.units > 0x7fffffffLL || plan.m_tiles > 0x7fffffff ||
      static_cast<long long>(desc->batch) * desc->n_kv_heads > 65535 || plan.splits > 65535)
    return ZARYA_ERR_UNSUPPORTED;
  if (plan.bytes > 0) {
    if (workspace == nullptr || workspace_bytes < plan.bytes ||
        (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
      return ZARYA_ERR_INVALID_ARG;
  }

  const int D = desc->head_dim, Hq = desc->n_q_heads, Hkv = desc->n_kv_heads, g = plan.g;
  CUtensorMap map_q, map_k, map_v;
  {
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(Hq),
                                static_cast<cuuint64_t>(desc->total_rows)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(D) * 2,
                                   static_cast<cuuint64_t>(Hq) * D * 2};
    const cuuint32_t box[3] = {64, static_cast<cuuint32_t>(g),
                               static_cast<cuuint32_t>(kBlockM / g)};
    if (encode(&map_q, const_cast<void*>(q), 3, dims, strides, box) != CUDA_SUCCESS)
      return cuda_fail("encoding the Q tensor map", cudaErrorInvalidValue);
  }
  {
    cuuint64_t dims[4], strides[3];
    cuuint32_t box[4];
    dims[0] = D;
    dims[1] = Hkv;
    strides[0] = static_cast<cuuint64_t>(D) * 2;
    strides[1] = static_cast<cuuint64_t>(Hkv) * D * 2;
    box[0] = 64;
    box[1] = 1;
    box[3] = 1;
    if (desc->page_size == 0) {
      dims[2] = desc->cache_capacity;
      dims[3] = desc->batch;
      strides[2] = static_cast<cuuint64_t>(desc->cache_capacity) * Hkv * D * 2;
      box[2] = kBlockN;
    } else {
      dims[2] = desc->page_size;
      dims[3] = desc->n_pages;
      strides[2] = static_cast<cuuint64_t>(desc->page_size) * Hkv * D * 2;
      box[2] = desc->page_size;
    }
    if (encode(&map_k, const_cast<void*>(k_cache), 4, dims, strides, box) != CUDA_SUCCESS ||
        encode(&map_v, const_cast<void*>(v_cache), 4, dims, strides, box) != CUDA_SUCCESS)
      return cuda_fail("encoding the K/V tensor maps", cudaErrorInvalidValue);
  }

  TcParams p{};
  p.cache_lens = cache_lens;
  p.page_table = page_table;
  p.n_slots = n_slots;
  p.slot_len = slot_len;
  p.mask_mode = mask_mode;
  p.q_row_offsets = desc->q_row_offsets;
  p.out = out;
  if (plan.bytes > 0) {
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    p.ws_o = reinterpret_cast<float*>(ws);
    p.ws_lse = reinterpret_cast<float*>(ws + plan.off_lse);
    p.ws_count = reinterpret_cast<int32_t*>(ws + plan.off_cnt);
  }
  p.err = err;
  p.B = desc->batch;
  p.Hq = Hq;
  p.Hkv = Hkv;
  p.g = g;
  p.max_rows = desc->max_rows;
  p.total_rows = desc->total_rows;
  p.capacity = desc->cache_capacity;
  p.page_size = desc->page_size;
  p.max_pages = max_pages;
  p.n_pages = desc->n_pages;
  p.m_tiles = plan.m_tiles;
  p.splits = plan.splits;
  p.cluster = (plan.splits > 1 && plan.splits <= kMaxClusterSplits) ? 1 : 0;
  p.pair = plan.pair;
  p.items = plan.items;
  p.perm = plan.sched ? static_cast<const int32_t*>(workspace) : nullptr;
  p.scale_log2 = scale * 1.4426950408889634f;
  p.wait_ns = desc->wait_limit_us > 0 ? static_cast<uint64_t>(desc->wait_limit_us) * 1000ull
                                       : 2000000000ull;
  p.debug_stall = (desc->debug_flags & ZARYA_DEBUG_STALL) ? 1 : 0;
  p.k_new = k_new;
  p.v_new = v_new;
  p.k_cache = const_cast<void*>(k_cache);
  p.v_cache = const_cast<void*>(v_cache);
  if (plan.sched) {
    ce = launch_schedule(p, stream);
    if (ce != cudaSuccess) return cuda_fail("launching schedule_kernel", ce);
  }
  ce = launch_slot_attn_tc(map_q, map_k, map_v, p, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching slot_attn_tc_kernel", ce);
}

zarya_status kv_append_impl(const void* k_new, const void* v_new, const int32_t* accept_len,
                            void* k_cache, void* v_cache, const int32_t* cache_lens,
                            int32_t* new_lens, const int32_t* page_table, bool commit,
                            const zarya_attn_desc* desc, zarya_stream_t stream_) {
  zarya_status st = check_desc(desc);
  if (st != ZARYA_OK) return st;
  // accept_len == nullptr (internal use only): copy every block row
  if (!k_new || !v_new || !k_cache || !v_cache || !cache_lens) return ZARYA_ERR_INVALID_ARG;
  if (commit && !new_lens) return ZARYA_ERR_INVALID_ARG;
  if ((desc->page_size > 0) != (page_table != nullptr)) return ZARYA_ERR_INVALID_ARG;
  if (!aligned16(k_new) || !aligned16(v_new) || !aligned16(k_cache) || !aligned16(v_cache))
    return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, k_new);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  const int eb = desc->dtype == ZARYA_BF16 ? 2 : 4;
  AppendParams p{};
  p.k_new = k_new;
  p.v_new = v_new;
  p.accept_len = accept_len;
  p.k_cache = k_cache;
  p.v_cache = v_cache;
  p.cache_lens = cache_lens;
  p.new_lens = new_lens;
  p.page_table = page_table;
  p.q_row_offsets = desc->q_row_offsets;
  p.err = err;
  p.B = desc->batch;
  p.row_bytes = desc->n_kv_heads * desc->head_dim * eb;
  p.max_rows = desc->max_rows;
  p.total_rows = desc->total_rows;
  p.capacity = desc->cache_capacity;
  p.page_size = desc->page_size;
  p.max_pages = desc->page_size > 0 ? desc->cache_capacity / desc->page_size : 0;
  p.n_pages = desc->n_pages;
  if (desc->batch > 65535) return ZARYA_ERR_UNSUPPORTED;
  ce = launch_kv_append(p, commit, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the append kernel", ce);
}

zarya_status check_sample_desc(const zarya_sample_desc* d) {
  if (d == nullptr) return ZARYA_ERR_INVALID_ARG;
  if (d->batch < 1 || d->vocab < 1 || d->max_slots < 1 || d->total_rows < 1)
    return ZARYA_ERR_INVALID_ARG;
  if (d->dtype != ZARYA_BF16 && d->dtype != ZARYA_FP32) return ZARYA_ERR_INVALID_ARG;
  if (d->reserved != 0 || d->reserved2 != 0) return ZARYA_ERR_INVALID_ARG;
  const int eb = d->dtype == ZARYA_BF16 ? 2 : 4;
  if (d->row_stride < d->vocab || (d->row_stride * eb) % 16 != 0) return ZARYA_ERR_INVALID_ARG;
  if (!(d->temperature >= 0.f) || std::isinf(d->temperature)) return ZARYA_ERR_INVALID_ARG;
  if (std::isnan(d->slot_threshold) || std::isnan(d->token_threshold))
    return ZARYA_ERR_INVALID_ARG;
  if (d->row_offsets == nullptr) return ZARYA_ERR_INVALID_ARG;
  if (static_cast<long long>(d->batch) * d->max_slots > 0x7fffffffLL) return ZARYA_ERR_UNSUPPORTED;
  return ZARYA_OK;
}

}  // namespace

zarya_status zarya_draft_select(const void* logits, const int32_t* n_slots,
                                const int32_t* slot_len, int32_t* draft_tokens,
                                float* draft_prob, float* slot_conf, uint8_t* slot_selected,
                                int32_t* n_selected, int32_t* verify_row_offsets,
                                int32_t* verify_src_rows, int32_t* verify_tokens,
                                const zarya_sample_desc* desc, zarya_stream_t stream_) {
  zarya_status st = check_sample_desc(desc);
  if (st != ZARYA_OK) return st;
  if (!logits || !n_slots || !slot_len || !draft_tokens || !draft_prob || !slot_conf ||
      !slot_selected || !n_selected || !verify_row_offsets || !verify_src_rows || !verify_tokens)
    return ZARYA_ERR_INVALID_ARG;
  if (!aligned16(logits)) return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, logits);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  const SampleCall c{logits, n_slots, slot_len, desc, sm_count()};
  const DraftOutputs o{draft_tokens, draft_prob,         slot_conf,       slot_selected,
                       n_selected,   verify_row_offsets, verify_src_rows, verify_tokens};
  ce = launch_draft_select(c, o, err, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the draft-select kernels", ce);
}

zarya_status zarya_verify_accept(const void* logits, const int32_t* tokens,
                                 const int32_t* n_slots, const int32_t* slot_len,
                                 float* token_prob, int32_t* slot_accept, int32_t* accept_len,
                                 const zarya_sample_desc* desc, zarya_stream_t stream_) {
  zarya_status st = check_sample_desc(desc);
  if (st != ZARYA_OK) return st;
  if (!logits || !tokens || !n_slots || !slot_len || !token_prob || !slot_accept || !accept_len)
    return ZARYA_ERR_INVALID_ARG;
  if (!aligned16(logits)) return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, logits);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  const SampleCall c{logits, n_slots, slot_len, desc, sm_count()};
  ce = launch_verify_accept(c, tokens, token_prob, slot_accept, accept_len, err, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the verify-accept kernels", ce);
}

zarya_status zarya_slot_attn(const void* q, const void* k_cache, const void* v_cache,
                             const int32_t* cache_lens, const int32_t* page_table,
                             const int32_t* n_slots, const int32_t* slot_len,
                             const int32_t* mask_mode, void* out, void* workspace,
                             size_t workspace_bytes, const zarya_attn_desc* desc,
                             zarya_stream_t stream) {
  return slot_attn_impl(q, nullptr, nullptr, k_cache, v_cache, cache_lens, page_table, n_slots,
                        slot_len, mask_mode, out, workspace, workspace_bytes, desc, stream);
}

zarya_status zarya_slot_attn_staged(const void* q, const void* k_new, const void* v_new,
                                    void* k_cache, void* v_cache, const int32_t* cache_lens,
                                    const int32_t* page_table, const int32_t* n_slots,
                                    const int32_t* slot_len, const int32_t* mask_mode, void* out,
                                    void* workspace, size_t workspace_bytes,
                                    const zarya_attn_desc* desc, zarya_stream_t stream) {
  if (!k_new || !v_new) return ZARYA_ERR_INVALID_ARG;
  return slot_attn_impl(q, k_new, v_new, k_cache, v_cache, cache_lens, page_table, n_slots,
                        slot_len, mask_mode, out, workspace, workspace_bytes, desc, stream);
}

zarya_status zarya_kv_append(const void* k_new, const void* v_new, const int32_t* accept_len,
                             void* k_cache, void* v_cache, int32_t* cache_lens,
                             const int32_t* page_table, int32_t flags,
                             const zarya_attn_desc* desc, zarya_stream_t stream) {
  if (flags != ZARYA_APPEND_STAGE && flags != ZARYA_APPEND_COMMIT) return ZARYA_ERR_INVALID_ARG;
  if (!accept_len) return ZARYA_ERR_INVALID_ARG;
  const bool commit = flags == ZARYA_APPEND_COMMIT;
  return kv_append_impl(k_new, v_new, accept_len, k_cache, v_cache, cache_lens,
                        commit ? cache_lens : nullptr, page_table, commit, desc, stream);
}

zarya_status zarya_kv_append_commit_to(const void* k_new, const void* v_new,
                                       const int32_t* accept_len, void* k_cache, void* v_cache,
                                       const int32_t* cache_lens, int32_t* new_lens,
                                       const int32_t* page_table, const zarya_attn_desc* desc,
                                       zarya_stream_t stream) {
  if (!accept_len) return ZARYA_ERR_INVALID_ARG;
  return kv_append_impl(k_new, v_new, accept_len, k_cache, v_cache, cache_lens, new_lens,
                        page_table, true, desc, stream);
}

zarya_status zarya_kv_commit_staged(const int32_t* accept_len, const int32_t* cache_lens,
                                    int32_t* new_lens, const zarya_attn_desc* desc,
                                    zarya_stream_t stream_) {
  zarya_status st = check_desc(desc);
  if (st != ZARYA_OK) return st;
  if (!accept_len || !cache_lens || !new_lens) return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, cache_lens);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  AppendParams p{};
  p.accept_len = accept_len;
  p.cache_lens = cache_lens;
  p.new_lens = new_lens;
  p.q_row_offsets = desc->q_row_offsets;
  p.err = err;
  p.B = desc->batch;
  p.max_rows = desc->max_rows;
  p.total_rows = desc->total_rows;
  p.capacity = desc->cache_capacity;
  ce = launch_commit_lens(p, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the commit kernel", ce);
}

zarya_status zarya_sample_rows(const void* logits, int32_t* tokens, float* prob,
                               const zarya_sample_desc* desc, zarya_stream_t stream_) {
  zarya_status st = check_sample_desc(desc);
  if (st != ZARYA_OK) return st;
  if (!logits || !tokens || !prob || !aligned16(logits)) return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, logits);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  const SampleCall c{logits, nullptr, nullptr, desc, sm_count()};
  ce = launch_sample_rows(c, tokens, prob, err, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the row-sampling kernel", ce);
}

zarya_status zarya_repetition_penalty(void* logits, const int32_t* hist_offsets,
                                      const int32_t* hist_tokens, int32_t n_hist, float penalty,
                                      const zarya_sample_desc* desc, zarya_stream_t stream_) {
  zarya_status st = check_sample_desc(desc);
  if (st != ZARYA_OK) return st;
  if (!logits || !hist_offsets || !aligned16(logits)) return ZARYA_ERR_INVALID_ARG;
  if (n_hist < 0 || (n_hist > 0 && !hist_tokens)) return ZARYA_ERR_INVALID_ARG;
  if (!(penalty > 0.f) || std::isinf(penalty)) return ZARYA_ERR_INVALID_ARG;
  if (static_cast<size_t>((desc->vocab + 31) / 32) * 4 > 200 * 1024) return ZARYA_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, logits);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  PenaltyParams p{};
  p.logits = logits;
  p.row_offsets = desc->row_offsets;
  p.hist_offsets = hist_offsets;
  p.hist_tokens = hist_tokens;
  p.err = err;
  p.B = desc->batch;
  p.V = desc->vocab;
  p.rows = desc->total_rows;
  p.n_hist = n_hist;
  p.row_stride = desc->row_stride;
  p.penalty = penalty;
  p.bf16 = desc->dtype == ZARYA_BF16 ? 1 : 0;
  ce = launch_penalty(p, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the repetition-penalty kernel", ce);
}

zarya_status zarya_top_p(void* logits, float top_p, const zarya_sample_desc* desc,
                         zarya_stream_t stream_) {
  zarya_status st = check_sample_desc(desc);
  if (st != ZARYA_OK) return st;
  if (!logits || !aligned16(logits)) return ZARYA_ERR_INVALID_ARG;
  if (!(top_p > 0.f)) return ZARYA_ERR_INVALID_ARG;   // also NaN
  if (desc->vocab > kNucleusMaxVocab) return ZARYA_ERR_UNSUPPORTED;
  if (top_p >= 1.f) return ZARYA_OK;                  // the nucleus is the whole vocabulary
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, logits);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  NucleusParams p{};
  p.logits = logits;
  p.row_offsets = desc->row_offsets;
  p.B = desc->batch;
  p.V = desc->vocab;
  p.rows = desc->total_rows;
  p.row_stride = desc->row_stride;
  p.k2 = desc->temperature > 0.f ? 1.4426950408889634f / desc->temperature : 1.4426950408889634f;
  p.top_p = top_p;
  p.bf16 = desc->dtype == ZARYA_BF16 ? 1 : 0;
  ce = launch_nucleus(p, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the top_p kernel", ce);
}

zarya_status zarya_mode_a_budget(const int32_t* n_masked, int32_t batch, int32_t T, float alpha0,
                                 uint64_t seed, uint64_t offset, int32_t max_steps,
                                 int32_t* counts, int32_t* n_steps, zarya_stream_t stream_) {
  if (!n_masked || !counts || !n_steps || batch < 1 || max_steps < 1 || T < 0)
    return ZARYA_ERR_INVALID_ARG;
  if (!(alpha0 >= 0.f && alpha0 <= 1.f)) return ZARYA_ERR_INVALID_ARG;
  if (static_cast<long long>(batch) * max_steps > 0x7fffffffLL) return ZARYA_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, n_masked);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  ModeAParams p{};
  p.n_masked = n_masked;
  p.counts = counts;
  p.n_steps = n_steps;
  p.err = err;
  p.B = batch;
  p.T = T;
  p.max_steps = max_steps;
  p.alpha0 = alpha0;
  p.key0 = static_cast<uint32_t>(seed);
  p.key1 = static_cast<uint32_t>(seed >> 32);
  p.ctr3 = static_cast<uint32_t>(offset);
  ce = launch_mode_a_budget(p, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the budget kernel", ce);
}

zarya_status zarya_reorder(const int32_t* tokens, const uint8_t* is_masked,
                           const uint32_t* order_key, const int32_t* lens, int32_t batch,
                           int32_t max_len, int32_t* perm, int32_t* tokens_out,
                           int32_t* n_unmasked, zarya_stream_t stream_) {
  if (!tokens || !is_masked || !lens || !perm || !tokens_out || !n_unmasked)
    return ZARYA_ERR_INVALID_ARG;
  if (batch < 1 || max_len < 1 || static_cast<const void*>(tokens_out) == tokens)
    return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, tokens);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  ReorderParams p{};
  p.tokens = tokens;
  p.is_masked = is_masked;
  p.order_key = order_key;
  p.lens = lens;
  p.perm = perm;
  p.tokens_out = tokens_out;
  p.n_unmasked = n_unmasked;
  p.err = err;
  p.B = batch;
  p.max_len = max_len;
  ce = launch_reorder(p, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the reorder kernel", ce);
}

zarya_status zarya_restore(const int32_t* tokens, const int32_t* perm, const int32_t* lens,
                           int32_t batch, int32_t max_len, int32_t* tokens_out,
                           zarya_stream_t stream_) {
  if (!tokens || !perm || !lens || !tokens_out) return ZARYA_ERR_INVALID_ARG;
  if (batch < 1 || max_len < 1 || tokens_out == tokens) return ZARYA_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, tokens);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  ReorderParams p{};
  p.tokens = tokens;
  p.perm_in = perm;
  p.lens = lens;
  p.tokens_out = tokens_out;
  p.err = err;
  p.B = batch;
  p.max_len = max_len;
  ce = launch_restore(p, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the restore kernel", ce);
}

// Pointer attributes, or false (the runtime's error cleared) for a pointer the
// runtime cannot describe.
static bool pointer_kind(const void* p, cudaPointerAttributes* a) {
  *a = cudaPointerAttributes{};
  if (cudaPointerGetAttributes(a, p) != cudaSuccess) {
    cudaGetLastError();   // clear the error the query leaves behind
    return false;
  }
  return true;
}

// The address through which the current device reaches `p`: device memory of
// that device (or managed memory) as is, page-locked host memory through its
// mapping; nullptr for anything else (another device's memory, pageable host
// memory).
static const void* device_address(const void* p, const cudaPointerAttributes& a, int dev) {
  if (a.type == cudaMemoryTypeManaged) return p;
  if (a.type == cudaMemoryTypeDevice) return a.device == dev ? p : nullptr;
  if (a.type != cudaMemoryTypeHost) return nullptr;
  void* d = nullptr;
  if (cudaHostGetDevicePointer(&d, const_cast<void*>(p), 0) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return d;
}

zarya_status zarya_copy(const void* src, void* dst, size_t bytes, zarya_stream_t stream_) {
  if (!src || !dst) return ZARYA_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u)
    return ZARYA_ERR_INVALID_ARG;
  if (bytes == 0) return ZARYA_OK;
  cudaPointerAttributes as, ad;
  if (!pointer_kind(src, &as) || !pointer_kind(dst, &ad)) return ZARYA_ERR_INVALID_ARG;
  const auto on_device = [](const cudaPointerAttributes& a) {
    return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
  };
  if (!on_device(as) && !on_device(ad)) return ZARYA_ERR_INVALID_ARG;   // two host buffers
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce = select_device(stream, on_device(as) ? src : dst);
  if (ce != cudaSuccess) return cuda_fail("selecting the stream's device", ce);
  int dev = -1;
  if ((ce = cudaGetDevice(&dev)) != cudaSuccess) return cuda_fail("cudaGetDevice", ce);
  const void* s = device_address(src, as, dev);
  const void* d = device_address(dst, ad, dev);
  if (s == nullptr || d == nullptr) return ZARYA_ERR_INVALID_ARG;
  const uintptr_t a = reinterpret_cast<uintptr_t>(s), b = reinterpret_cast<uintptr_t>(d);
  if ((a | b) & 15u) return ZARYA_ERR_INVALID_ARG;
  if (a < b + bytes && b < a + bytes) return ZARYA_ERR_INVALID_ARG;   // overlapping ranges
  ce = launch_copy(s, const_cast<void*>(d), bytes, stream);
  return ce == cudaSuccess ? ZARYA_OK : cuda_fail("launching the copy kernel", ce);
}

zarya_status zarya_check_device_error(zarya_stream_t stream_, int32_t* code) {
  if (code) *code = 0;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_);
  cudaError_t ce;
  if (stream != nullptr) {
    int dev = -1, cur = -1;
    if ((ce = cudaStreamGetDevice(stream, &dev)) != cudaSuccess)
      return cuda_fail("cudaStreamGetDevice", ce);
    if ((ce = cudaGetDevice(&cur)) != cudaSuccess) return cuda_fail("cudaGetDevice", ce);
    if (cur != dev && (ce = cudaSetDevice(dev)) != cudaSuccess)
      return cuda_fail("cudaSetDevice", ce);
  }
  int* err = device_error_word(&ce);
  if (err == nullptr) return cuda_fail("looking up the device error word", ce);
  int host = 0;
  if ((ce = cudaStreamSynchronize(stream)) != cudaSuccess)
    return cuda_fail("cudaStreamSynchronize", ce);
  if ((ce = cudaMemcpyAsync(&host, err, sizeof(int), cudaMemcpyDeviceToHost, stream)) !=
      cudaSuccess)
    return cuda_fail("reading the device error word", ce);
  if ((ce = cudaMemsetAsync(err, 0, sizeof(int), stream)) != cudaSuccess)
    return cuda_fail("clearing the device error word", ce);
  if ((ce = cudaStreamSynchronize(stream)) != cudaSuccess)
    return cuda_fail("cudaStreamSynchronize", ce);
  if (code) *code = host;
  return host == 0 ? ZARYA_OK : ZARYA_ERR_DEVICE_FAULT;
}

const char* zarya_last_error(void) { return g_last_error; }

const char* zarya_status_string(zarya_status status) {
  switch (status) {
    case ZARYA_OK: return "ok";
    case ZARYA_ERR_INVALID_ARG: return "invalid argument";
    case ZARYA_ERR_UNSUPPORTED: return "unsupported configuration";
    case ZARYA_ERR_CUDA: return "CUDA error";
    case ZARYA_ERR_DEVICE_FAULT: return "device error word set";
  }
  return "unknown status";
}

int32_t zarya_version(void) { return kVersion; }

}  // extern "C"
