// Internal declarations shared by the library's translation units: kernel
// parameter blocks, launchers and the per-device error word.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "zarya.h"

namespace zarya {

// Tile geometry of the tensor-core path (bf16, D = 128).
constexpr int kBlockM = 128;  // packed (block row, query head) rows per CTA
constexpr int kBlockN = 128;  // keys per pipeline tile
constexpr int kHeadDim = 128;
// At most this many key splits of one tile merge inside a thread-block cluster
// (each split receives the rows it finishes from the others in its idle K ring).
constexpr int kMaxClusterSplits = 3;

// Parameters of the tensor-core slot-attention kernel (tensor maps travel as
// separate __grid_constant__ arguments).
struct TcParams {
  const int32_t* cache_lens;
  const int32_t* page_table;
  const int32_t* n_slots;
  const int32_t* slot_len;
  const int32_t* mask_mode;
  const int32_t* q_row_offsets;
  void* out;          // bf16 [total_rows, Hq, D]
  float* ws_o;        // [units, splits, kBlockM, D] fp32 partial outputs (normalised)
  float* ws_lse;      // [units, splits, kBlockM] log2-sum-exp of each partial
  int32_t* ws_count;  // [units] arrival counters of the workspace merge (zero between calls)
  int* err;           // device error word
  int B, Hq, Hkv, g;
  int max_rows, total_rows, capacity;
  int page_size, max_pages, n_pages;
  int m_tiles, splits;
  int cluster;        // 1: the splits of a tile form a cluster and merge through DSMEM
  int pair;           // 1: one CTA per pair of M-tiles (paged caches, no key split)
  // Longest-first dispatch (no key split, several waves): the CTA at linear
  // position pos serves KV head pos % Hkv of work item perm[pos / Hkv], item
  // i being (sequence i / items, M-tile or pair i % items); nullptr: the grid's
  // own order.
  const int32_t* perm;
  int items;          // work items per sequence (M-tiles, or pairs of them)
  float scale_log2;   // softmax scale * log2(e)
  uint64_t wait_ns;   // bound on every pipeline wait (global-timer nanoseconds)
  int debug_stall;    // 1: the MMA warp first waits on a barrier nothing completes
  // Staged attention: when k_new != nullptr, block row i of sequence b
  // (k_new / v_new row q_row_offsets[b] + i) is first written to cache
  // position P_b + i by the CTAs that read it.
  const void* k_new;  // bf16 [total_rows, Hkv, D] or nullptr
  const void* v_new;
  void* k_cache;      // bf16 cache (the tensor maps' base addresses)
  void* v_cache;
};

// Parameters of the fp32 CUDA-core path and of the append kernels.
struct SimtParams {
  const void* q;
  const void* k_cache;
  const void* v_cache;
  const int32_t* cache_lens;
  const int32_t* page_table;
  const int32_t* n_slots;
  const int32_t* slot_len;
  const int32_t* mask_mode;
  const int32_t* q_row_offsets;
  void* out;
  int* err;
  int B, Hq, Hkv, D;
  int max_rows, total_rows, capacity;
  int page_size, max_pages, n_pages;
  float scale;
};

struct AppendParams {
  const void* k_new;
  const void* v_new;
  const int32_t* accept_len;
  void* k_cache;
  void* v_cache;
  const int32_t* cache_lens;
  int32_t* new_lens;        // commit: receives cache_lens[b] + accept_len[b] (may alias cache_lens)
  const int32_t* page_table;
  const int32_t* q_row_offsets;
  int* err;
  int B, row_bytes;  // row_bytes = Hkv * D * element size (multiple of 16)
  int max_rows, total_rows, capacity;
  int page_size, max_pages, n_pages;
  int rows_per_block;       // block rows copied by one CTA (gridDim.x CTAs per sequence)
};

// Common inputs of the slot-selection and token-acceptance calls.
struct SampleCall {
  const void* logits;
  const int32_t* n_slots;
  const int32_t* slot_len;
  const zarya_sample_desc* desc;
  int sms;  // multiprocessors of the device (sizes the row split)
};

struct DraftOutputs {
  int32_t* draft_tokens;
  float* draft_prob;
  float* slot_conf;
  uint8_t* slot_selected;
  int32_t* n_selected;
  int32_t* verify_row_offsets;
  int32_t* verify_src_rows;
  int32_t* verify_tokens;
};

cudaError_t launch_draft_select(const SampleCall& c, const DraftOutputs& o, int* err,
                                cudaStream_t stream);
cudaError_t launch_verify_accept(const SampleCall& c, const int32_t* tokens, float* token_prob,
                                 int32_t* slot_accept, int32_t* accept_len, int* err,
                                 cudaStream_t stream);

// Dynamic shared memory of the tensor-core kernel.
size_t tc_smem_bytes();

// Most work items one dispatch order can sort (B x items).
constexpr int kMaxSchedItems = 4096;
// Writes p.perm: the work items sorted by cost (M-tiles x key tiles), largest first.
cudaError_t launch_schedule(const TcParams& p, cudaStream_t stream);

cudaError_t launch_slot_attn_tc(const CUtensorMap& map_q, const CUtensorMap& map_k,
                                const CUtensorMap& map_v, const TcParams& p,
                                cudaStream_t stream);
cudaError_t launch_slot_attn_f32(const SimtParams& p, cudaStream_t stream);
cudaError_t launch_kv_append(const AppendParams& p, bool commit, cudaStream_t stream);
// new_lens[b] = cache_lens[b] + accept_len[b] after the device checks of the
// append (the block's rows are already in the cache).
cudaError_t launch_commit_lens(const AppendParams& p, cudaStream_t stream);

// Bytes at the end of the attention workspace that hold the split counters
// (which must be zero before a call); 0 when the plan needs no workspace.
size_t workspace_counter_bytes(const zarya_attn_desc* desc);

// Launch configuration with programmatic stream serialisation enabled, so a
// kernel's set-up can overlap the tail of the kernel before it.
struct PdlLaunch {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[2];
  // cluster_x > 1: thread-block clusters of cluster_x CTAs along x.
  PdlLaunch(dim3 grid, dim3 block, size_t smem, cudaStream_t stream, unsigned cluster_x = 1)
      : cfg{}, attr{} {
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cluster_x > 1) {
      attr[1].id = cudaLaunchAttributeClusterDimension;
      attr[1].val.clusterDim.x = cluster_x;
      attr[1].val.clusterDim.y = 1;
      attr[1].val.clusterDim.z = 1;
      cfg.numAttrs = 2;
    }
  }
};

// Makes the device that owns `stream` (or, while it captures a graph or for
// the legacy default stream, the device that owns `ptr`) current.
cudaError_t select_device(cudaStream_t stream, const void* ptr);

// Records "what: <CUDA error string>" as this thread's last error message
// (zarya_last_error) and returns ZARYA_ERR_CUDA.
zarya_status cuda_fail(const char* what, cudaError_t e);

// Address of the error word on the current device (set-up once per device).
int* device_error_word(cudaError_t* status);

// Records `code` in the error word unless an earlier error is already there.
__device__ __forceinline__ void record_error(int* err, int code) {
  atomicCAS(err, 0, code);
}

}  // namespace zarya
