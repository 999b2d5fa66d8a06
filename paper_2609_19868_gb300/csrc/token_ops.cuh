// Declarations of the token-level kernels that sit around the attention
// step (row sampling of Mode A, the repetition penalty and top_p truncation
// of logits, reordering / restoration, Mode A planning) and of the SM copy
// kernel, shared by their translation units and the C ABI.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "internal.cuh"

namespace zarya {

cudaError_t launch_sample_rows(const SampleCall& c, int32_t* tokens, float* prob, int* err,
                               cudaStream_t stream);

// SM copy of `bytes` bytes between device addresses (device memory, or the
// device mapping of page-locked host memory); src and dst 16-byte aligned.
cudaError_t launch_copy(const void* src, void* dst, size_t bytes, cudaStream_t stream);

// Repetition penalty over logits rows, in place.
struct PenaltyParams {
  void* logits;                // [rows, row_stride] bf16 or fp32
  const int32_t* row_offsets;  // [B + 1] rows of each sequence
  const int32_t* hist_offsets; // [B + 1] history tokens of each sequence
  const int32_t* hist_tokens;  // [n_hist]
  int* err;
  int B, V, rows, n_hist;
  int64_t row_stride;          // elements
  float penalty;
  int bf16;
};

cudaError_t launch_penalty(const PenaltyParams& p, cudaStream_t stream);

// top_p truncation of logits rows, in place.
struct NucleusParams {
  void* logits;                // [rows, row_stride] bf16 or fp32
  const int32_t* row_offsets;  // [B + 1] rows of each sequence
  int B, V, rows;
  int64_t row_stride;          // elements
  float k2;                    // log2(e) / T (log2(e) at T = 0)
  float top_p;
  int bf16;
};

// The largest vocabulary the top_p kernel takes (its per-thread 32-bit mass
// sums stay below 2^32 up to it).
constexpr int kNucleusMaxVocab = 520192;
cudaError_t launch_nucleus(const NucleusParams& p, cudaStream_t stream);

// Reordering / restoration of [B, max_len] token rows.
struct ReorderParams {
  const int32_t* tokens;
  const uint8_t* is_masked;   // reorder
  const uint32_t* order_key;  // reorder, optional
  const int32_t* lens;
  const int32_t* perm_in;     // restore
  int32_t* perm;              // reorder
  int32_t* tokens_out;
  int32_t* n_unmasked;        // reorder
  int* err;
  int B, max_len;
};

cudaError_t launch_reorder(const ReorderParams& p, cudaStream_t stream);
cudaError_t launch_restore(const ReorderParams& p, cudaStream_t stream);

// Mode A mask-budget planning.
struct ModeAParams {
  const int32_t* n_masked;
  int32_t* counts;     // [B, max_steps]
  int32_t* n_steps;    // [B]
  int* err;
  int B, T, max_steps;
  float alpha0;
  uint32_t key0, key1, ctr3;
};

cudaError_t launch_mode_a_budget(const ModeAParams& p, cudaStream_t stream);

}  // namespace zarya
