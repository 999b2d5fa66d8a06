/*
 * zarya.h -- C ABI of the GB300 (sm_103a) slot-attention library.
 *
 * The library implements the per-layer attention step of Zarya's slotted
 * speculative decoding (Mode B, Sec. 5.2 of "Zarya: A Hybrid
 * Autoregressive--Masked Diffusion Language Model with Flexible Training and
 * Dual-Mode Inference") and the KV-cache update with accepted tokens that
 * gives the mode its full KV reuse (Sec. 5.2 step 7; Sec. 5.1 explains why the
 * reordered prefix cache stays valid under causal attention). Around it sit
 * the token-level steps of both inference modes: slot selection and token
 * acceptance (Sec. 5.2 steps 3-6), Mode A's reveal plan and per-step draws
 * (Sec. 5.1 steps 1 and 3) with the repetition penalty and top_p they honour
 * (Table 2), and the reordering / restoration of sequences (Sec. 5.1 steps 2
 * and 4, Sec. 5.2 steps 1 and 8).
 *
 * Notation: sequence b of a batch of B; committed prefix length
 * P_b = cache_lens[b]; the current block holds S_b = n_slots[b] slots of
 * L_b = slot_len[b] tokens, R_b = S_b * L_b query rows, placed right after the
 * prefix by the reordering step (Sec. 5.2 steps 1-2). Block row r = s*L_b + j
 * (slot s, offset j). Key index c < P_b is a prefix token; c >= P_b is block
 * row c - P_b, whose K/V must have been staged into the cache at positions
 * P_b .. P_b + R_b - 1 (zarya_kv_append with ZARYA_APPEND_STAGE) before
 * zarya_slot_attn runs.
 *
 * General rules for every entry point:
 *  - All array arguments are DEVICE pointers on the device that owns `stream`
 *    (the caller owns every buffer), except where a call says otherwise
 *    (zarya_copy also takes page-locked host buffers). Calls are asynchronous
 *    on `stream`; none blocks except zarya_check_device_error.
 *  - Host-side validation happens first; an invalid call returns a status and
 *    launches nothing. Nothing falls back to the CPU.
 *  - Errors that only the device can see (a page id out of range, a length
 *    beyond capacity, inconsistent row offsets, a pipeline wait that timed
 *    out) set a per-device error word; the affected work is skipped, never
 *    trapped. Read (and clear) it with zarya_check_device_error.
 *  - bf16 tensors use round-to-nearest-even on output; fp32 accumulation.
 *  - The library keeps per-device set-up for the life of the process: the
 *    device addresses of its error word and of the zarya_slot_attn_noalloc
 *    scratch, and kernel attributes. Do not call it on a device after
 *    cudaDeviceReset there: the cached addresses would point into the
 *    destroyed context.
 */
#ifndef ZARYA_H_
#define ZARYA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* zarya_stream_t;

typedef enum {
  ZARYA_OK = 0,
  ZARYA_ERR_INVALID_ARG = 1,   /* bad pointer, size, alignment or descriptor field */
  ZARYA_ERR_UNSUPPORTED = 2,   /* valid request this build does not implement */
  ZARYA_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed */
  ZARYA_ERR_DEVICE_FAULT = 4   /* the device error word was set (see below) */
} zarya_status;

/* Mask of one sequence's block (Sec. 5.2). */
typedef enum {
  /* Draft pass (step 3, inter-slot diffusion selection): every block row sees
   * the whole prefix and the whole block: visible(c) <=> c < P_b + R_b. */
  ZARYA_MASK_BIDIR_BLOCK = 0,
  /* Verification pass (step 6, intra-slot autoregressive infilling): causal
   * over the reordered, flattened sequence: visible(c) <=> c < P_b + r + 1. */
  ZARYA_MASK_SLOT_CAUSAL = 1,
  /* Verification of several selected slots in one pass, each on its own
   * (step 6 with parallel slots): block row r = s*L_b + j sees the prefix and
   * rows s*L_b .. r of its own slot:
   * visible(c) <=> c < P_b or P_b + s*L_b <= c <= P_b + r. */
  ZARYA_MASK_SLOT_INDEPENDENT = 2
} zarya_mask_mode;

typedef enum { ZARYA_BF16 = 0, ZARYA_FP32 = 1 } zarya_dtype;

/* zarya_kv_append flags */
#define ZARYA_APPEND_STAGE 0   /* write rows at P_b.., leave cache_lens unchanged */
#define ZARYA_APPEND_COMMIT 1  /* write rows at P_b.., then cache_lens[b] += accept_len[b] */

/* Device error word values (zarya_check_device_error's *code). */
#define ZARYA_DEVERR_NONE 0
#define ZARYA_DEVERR_PAGE_ID 1        /* page_table entry outside [0, n_pages) */
#define ZARYA_DEVERR_ROWS 2           /* R_b > max_rows, or q_row_offsets inconsistent with R_b */
#define ZARYA_DEVERR_CAPACITY 3       /* P_b + rows would pass cache_capacity */
#define ZARYA_DEVERR_ACCEPT 4         /* accept_len[b] outside [0, R_b] */
#define ZARYA_DEVERR_TIMEOUT 5        /* a pipeline wait gave up (no progress for
                                         desc->wait_limit_us, 2 s by default) */
#define ZARYA_DEVERR_MASK_MODE 6      /* mask_mode[b] not a zarya_mask_mode */
#define ZARYA_DEVERR_TOKEN 7          /* a verification token outside [0, vocab) */
#define ZARYA_DEVERR_PERM 8           /* a permutation entry outside [0, lens[b]) */

/* Shapes and host-known bounds shared by both calls. */
typedef struct {
  int32_t batch;           /* B >= 1 */
  int32_t n_q_heads;       /* Hq; Hq % Hkv == 0 (query head h reads KV head h / (Hq/Hkv)) */
  int32_t n_kv_heads;      /* Hkv */
  int32_t head_dim;        /* D: 128 for bf16; 32..256 (multiple of 32) for fp32 */
  int32_t dtype;           /* zarya_dtype of q, caches, k_new/v_new and out */
  int32_t page_size;       /* 0: contiguous cache [B, cache_capacity, Hkv, D];
                              else paged cache [n_pages, page_size, Hkv, D] with a page table
                              [B, cache_capacity / page_size]; bf16 needs 16, 32, 64 or 128 */
  int32_t cache_capacity;  /* tokens per sequence (paged: max pages per sequence * page_size) */
  int32_t n_pages;         /* paged: pages in the pool (page ids must lie in [0, n_pages)) */
  int32_t max_rows;        /* upper bound on R_b over the batch (sizes the grid, no host sync) */
  int32_t total_rows;      /* rows of q / out / k_new / v_new = q_row_offsets[B] */
  int32_t max_kv_len;      /* upper bound on P_b + R_b (0: use cache_capacity); sizes splits */
  int32_t kv_splits;       /* 0: choose automatically; n > 0: split each key range n ways */
  float scale;             /* softmax scale; 0 means 1 / sqrt(D) */
  const int32_t* q_row_offsets; /* device [B + 1]: first row of sequence b in q / out /
                                   k_new; q_row_offsets[b+1] - q_row_offsets[b] == R_b */
  int32_t wait_limit_us;   /* bound on every pipeline wait of the tensor-core attention kernel,
                              in microseconds of global time; 0 = 2,000,000 (2 s). A wait that
                              runs out sets ZARYA_DEVERR_TIMEOUT and its CTA unwinds (lets its
                              own copies and MMAs finish, frees its tensor memory, writes no
                              output). A failure-detection knob: normal waits last microseconds. */
  int32_t debug_flags;     /* 0 in normal use; ZARYA_DEBUG_STALL tests the timeout path */
} zarya_attn_desc;

/* zarya_attn_desc.debug_flags: the tensor-core attention kernel's MMA warp
 * first waits on a barrier that nothing completes, so that wait runs out after
 * wait_limit_us and the launch unwinds with ZARYA_DEVERR_TIMEOUT, leaving the
 * device usable (used by tests of the failure path; with kv_splits = 1 or
 * more than 3, i.e. no thread-block cluster merge). */
#define ZARYA_DEBUG_STALL 1

/*
 * Bytes of scratch memory zarya_slot_attn needs for `desc` (0 if it needs
 * none). The workspace holds split-KV partial results and per-tile arrival
 * counters (more than 3 key splits), or the dispatch order of the work tiles
 * (slot_attn_pair_kernel taking several waves of CTAs). It must be zero-filled
 * once before its first use; every call leaves the counters at zero again, so
 * it can be reused by later calls on the same stream. After a call that set
 * the device error word, zero it again.
 * Returns 0 as well when desc is invalid (zarya_slot_attn will reject it).
 */
size_t zarya_slot_attn_workspace_size(const zarya_attn_desc* desc);

/*
 * Name of the kernel zarya_slot_attn launches for `desc` on the current
 * device (for profilers and reports): "slot_attn_tc_kernel" (one M-tile of
 * 128 packed rows per CTA, key range split across CTAs where that pays),
 * "slot_attn_pair_kernel" (paged caches whose M-tile pairs fill the GPU: two
 * M-tiles per CTA sharing every K/V tile), "slot_attn_f32_kernel" (fp32), or
 * "none" for a descriptor zarya_slot_attn would reject. A static string; no
 * device work.
 */
const char* zarya_slot_attn_kernel(const zarya_attn_desc* desc);

/*
 * Kernels one zarya_slot_attn call launches for `desc` on the current device:
 * 2 when the plan sorts its work tiles first (slot_attn_pair_kernel taking
 * several waves of CTAs: a one-CTA kernel writes the longest-first dispatch
 * order into the workspace, then the attention kernel follows it), else 1;
 * 0 for a descriptor zarya_slot_attn would reject. zarya_slot_attn_staged
 * with fp32 launches one more (the staging append). No device work.
 */
int32_t zarya_slot_attn_launches(const zarya_attn_desc* desc);

/*
 * Slot attention (Sec. 5.2 steps 3 and 6): for every sequence b, query head
 * h and block row r < R_b,
 *   out[q_row_offsets[b] + r, h, :] =
 *     sum_{c visible} softmax_c(scale * q[q_row_offsets[b] + r, h, :] . k_c) v_c
 * with k_c / v_c the cache entries of token c of sequence b at KV head
 * h / (Hq / Hkv), and visibility given by mask_mode[b] (zarya_mask_mode).
 *
 *  q          [total_rows, Hq, D]                     (read)
 *  k_cache,   contiguous [B, cache_capacity, Hkv, D]  (read; positions
 *  v_cache    or paged [n_pages, page_size, Hkv, D]    0 .. P_b + R_b - 1 used)
 *  cache_lens [B] int32: P_b, the committed prefix (block K/V already staged after it)
 *  page_table [B, cache_capacity / page_size] int32, or NULL for a contiguous cache
 *  n_slots, slot_len, mask_mode: [B] int32 each
 *  out        [total_rows, Hq, D]                     (written; rows of each
 *                                                      sequence only)
 *  workspace  zarya_slot_attn_workspace_size(desc) bytes (may be NULL when that is 0)
 * Pointers q, caches and out must be 16-byte aligned. q/out rows that belong
 * to no sequence are not written.
 */
zarya_status zarya_slot_attn(const void* q, const void* k_cache, const void* v_cache,
                             const int32_t* cache_lens, const int32_t* page_table,
                             const int32_t* n_slots, const int32_t* slot_len,
                             const int32_t* mask_mode, void* out, void* workspace,
                             size_t workspace_bytes, const zarya_attn_desc* desc,
                             zarya_stream_t stream);

/*
 * The block's own K/V staged and attended in one launch: exactly
 * zarya_kv_append(k_new, v_new, <R_b for every b>, ..., ZARYA_APPEND_STAGE)
 * followed by zarya_slot_attn(...) on the same stream (Sec. 5.2 step 3: the
 * block attends over the cached prefix plus itself, its K/V coming from the
 * same forward pass). k_new / v_new are [total_rows, Hkv, D] like the append's;
 * block row i of sequence b is written to cache position P_b + i (through the
 * page table when paged) and cache_lens is left alone. On the tensor-core path
 * the CTAs that read a block row copy it into the cache themselves just before
 * loading it, so the copy overlaps the streaming of the prefix. Arguments,
 * workspace and errors as zarya_slot_attn; k_new / v_new must be non-NULL and
 * 16-byte aligned.
 */
zarya_status zarya_slot_attn_staged(const void* q, const void* k_new, const void* v_new,
                                    void* k_cache, void* v_cache, const int32_t* cache_lens,
                                    const int32_t* page_table, const int32_t* n_slots,
                                    const int32_t* slot_len, const int32_t* mask_mode, void* out,
                                    void* workspace, size_t workspace_bytes,
                                    const zarya_attn_desc* desc, zarya_stream_t stream);

/*
 * zarya_slot_attn without a workspace argument, for callers that cannot
 * allocate device memory at the point where they run attention: a serving
 * engine that has already given all of HBM to its own cache pool, a host
 * application whose plug-ins may not allocate device memory, or a decode loop
 * that cannot afford cudaMalloc / cudaFree (both can synchronise the device).
 * The paper has no counterpart; this is a deployment convenience.
 *
 * Same arguments, results and errors as zarya_slot_attn, minus workspace.
 * The split-KV scratch is a 16 MiB array inside the library, reserved on
 * every GPU that loads it until the process exits; this call allocates
 * nothing. A descriptor whose split plan needs more than 16 MiB
 * (zarya_slot_attn_workspace_size(desc) > 16 MiB) is rejected with
 * ZARYA_ERR_UNSUPPORTED and nothing is launched; set desc->kv_splits = 1
 * (no scratch needed) or use zarya_slot_attn with a workspace.
 * The first call on each device looks up the scratch address on that device
 * (a one-time set-up step); make that first call before any stream capture.
 * Every call on a device shares the one scratch array, which keeps what the
 * last call left: each call zeroes the part that must start at zero (the
 * split arrival counters) on `stream` before its kernel runs, so calls in
 * order on one stream are safe, but calls that overlap on the GPU (different
 * streams, or different threads) race on the scratch and give wrong results.
 */
zarya_status zarya_slot_attn_noalloc(const void* q, const void* k_cache, const void* v_cache,
                                     const int32_t* cache_lens, const int32_t* page_table,
                                     const int32_t* n_slots, const int32_t* slot_len,
                                     const int32_t* mask_mode, void* out,
                                     const zarya_attn_desc* desc, zarya_stream_t stream);

/*
 * KV-cache update with accepted tokens (Sec. 5.2 step 7): for every sequence
 * b and i < accept_len[b], row q_row_offsets[b] + i of k_new / v_new
 * ([total_rows, Hkv, D], the block rows in reordered order, accepted tokens
 * first) is copied bit for bit to cache position P_b + i (through the page
 * table when paged). With ZARYA_APPEND_COMMIT, cache_lens[b] then advances by
 * accept_len[b]; with ZARYA_APPEND_STAGE it is left alone (used to stage a
 * block's own K/V before its attention pass). 0 <= accept_len[b] <= R_b and
 * P_b + accept_len[b] <= cache_capacity are checked on the device; a sequence
 * that fails is skipped and the error word set. Nothing else in the caches
 * changes.
 */
zarya_status zarya_kv_append(const void* k_new, const void* v_new, const int32_t* accept_len,
                             void* k_cache, void* v_cache, int32_t* cache_lens,
                             const int32_t* page_table, int32_t flags,
                             const zarya_attn_desc* desc, zarya_stream_t stream);

/*
 * The ZARYA_APPEND_COMMIT form of zarya_kv_append with the advanced lengths
 * going to a second array: the same rows are copied to positions
 * cache_lens[b] + i, and new_lens[b] (device [B]) receives
 * cache_lens[b] + accept_len[b] for every sequence that passed the device
 * checks (others keep their new_lens entry and set the error word).
 * cache_lens is only read. new_lens may be cache_lens itself, which is then
 * exactly zarya_kv_append(..., ZARYA_APPEND_COMMIT, ...). A caller that keeps
 * the lengths of consecutive steps in two arrays (ping-pong) needs no copy
 * between steps. Not a step of the paper's method, only a form of step 7.
 */
zarya_status zarya_kv_append_commit_to(const void* k_new, const void* v_new,
                                       const int32_t* accept_len, void* k_cache, void* v_cache,
                                       const int32_t* cache_lens, int32_t* new_lens,
                                       const int32_t* page_table, const zarya_attn_desc* desc,
                                       zarya_stream_t stream);

/*
 * Step 7 for a block whose rows are already in the cache: after the
 * verification pass staged its block (zarya_slot_attn_staged, or
 * zarya_kv_append with ZARYA_APPEND_STAGE, from the same k_new / v_new whose
 * accepted rows come first), rows 0 .. accept_len[b] - 1 of the block already
 * sit at positions P_b .. P_b + accept_len[b] - 1, so the commit only
 * advances the length: new_lens[b] = cache_lens[b] + accept_len[b]. No cache
 * byte moves; afterwards the cache holds exactly what zarya_kv_append_commit_to
 * would leave in positions below new_lens[b]. accept_len, cache_lens: device
 * [B] (read); new_lens: device [B] (written; may be cache_lens). The device
 * checks and error behaviour are those of zarya_kv_append (a sequence that
 * fails keeps its new_lens entry and sets the error word). Waits for the
 * work queued before it on `stream`.
 */
zarya_status zarya_kv_commit_staged(const int32_t* accept_len, const int32_t* cache_lens,
                                    int32_t* new_lens, const zarya_attn_desc* desc,
                                    zarya_stream_t stream);

/* ------------------------------------------------------------------------
 * Slot selection and token acceptance (Sec. 5.2 steps 3-6).
 *
 * The draft pass (step 3, ZARYA_MASK_BIDIR_BLOCK attention) yields logits for
 * every block row. zarya_draft_select draws one token per row, takes each
 * slot's confidence as the probability of the token drawn at its first row
 * (step 3), and selects the slots to verify (step 5): those whose confidence
 * exceeds slot_threshold, or, when none does, the single most confident one.
 * It lays out the verification block: the selected slots' rows, in slot
 * order, packed densely per sequence (n_selected[b] * L_b rows each), which is
 * the q / k_new row layout of the verification attention pass.
 *
 * The verification pass (step 6, ZARYA_MASK_SLOT_CAUSAL or
 * ZARYA_MASK_SLOT_INDEPENDENT attention over the verification block) yields
 * logits for those rows. zarya_verify_accept takes the probability of each
 * drafted token and accepts tokens while it exceeds token_threshold: per
 * verified slot its accepted prefix, and over the whole verification block
 * the accepted prefix length accept_len[b], which zarya_kv_append commits
 * (step 7).
 *
 * Definitions used by both calls:
 *  - Row probability of token t: softmax(x / T)[t] over the V logits x of the
 *    row (softmax(x) when T = 0), computed in fp32.
 *  - Draw (steps 3-4): T = 0: argmax of x. T > 0: Gumbel-max sampling, the
 *    argmax of x / T + g_v with g_v standard Gumbel noise. Ties go to the
 *    lowest vocabulary index; comparisons of probabilities with thresholds
 *    are strict.
 *  - Noise: g_v of logits row `row` comes from Philox4x32-10 (Salmon et al.,
 *    SC'11) with key (seed low word, seed high word) and counter
 *    (v / 4, row, offset low word, offset high word); word v % 4 of the
 *    output is w, u = fl32(fl32(w) * 2^-32 + 2^-33) in (0, 1],
 *    E = -log1p(-u), g_v = -log(E), in fp32.
 *  - Logits rows: row r of the batch starts at element r * row_stride of
 *    `logits` (bf16 or fp32, 16-byte aligned). Sequence b owns rows
 *    row_offsets[b] .. row_offsets[b+1] - 1, which must number
 *    n_slots[b] * slot_len[b] (device check: ZARYA_DEVERR_ROWS, and the
 *    sequence is skipped); slot s of sequence b is its rows s*L_b .. s*L_b +
 *    L_b - 1. Rows outside every sequence are not read.
 */
typedef struct {
  int32_t batch;            /* B >= 1 */
  int32_t vocab;            /* V >= 1 */
  int32_t dtype;            /* zarya_dtype of the logits */
  int32_t max_slots;        /* >= every S_b; row length of slot_conf, slot_selected, slot_accept */
  int32_t total_rows;       /* rows of the logits buffer and of the per-row outputs;
                               >= row_offsets[B] */
  int32_t reserved;         /* must be 0 */
  int64_t row_stride;       /* elements from one logits row to the next: >= vocab, and
                               row_stride * element size a multiple of 16 bytes */
  float temperature;        /* T >= 0 (finite); 0 draws the argmax */
  float slot_threshold;     /* step 5 */
  float token_threshold;    /* step 6 */
  uint32_t reserved2;       /* must be 0 */
  uint64_t seed;            /* Philox key */
  uint64_t offset;          /* Philox counter words 2-3; a new value gives fresh noise */
  const int32_t* row_offsets; /* device [B + 1], non-decreasing */
} zarya_sample_desc;

/*
 * Steps 3-5. Inputs: logits [total_rows, row_stride]; n_slots, slot_len
 * device [B] (S_b, L_b >= 1, S_b <= max_slots). Outputs (device, written):
 *  draft_tokens       [total_rows] int32   drawn token of every block row
 *  draft_prob         [total_rows] float   its probability
 *  slot_conf          [B, max_slots] float confidence of slot s (0 for s >= S_b)
 *  slot_selected      [B, max_slots] uint8 1 if slot s is selected
 *  n_selected         [B] int32            selected slots (>= 1 for a valid sequence)
 *  verify_row_offsets [B + 1] int32        verification layout: running sum of
 *                                          n_selected[b] * L_b (starts at 0)
 *  verify_src_rows    [total_rows] int32   verification row k -> the draft row it
 *                                          verifies; -1 from verify_row_offsets[B] on
 *  verify_tokens      [total_rows] int32   the token drafted at that row; -1 after
 * Per-row outputs of rows outside every sequence are not written. A sequence
 * that fails the device checks gets n_selected[b] = 0 (no verification rows).
 */
zarya_status zarya_draft_select(const void* logits, const int32_t* n_slots,
                                const int32_t* slot_len, int32_t* draft_tokens,
                                float* draft_prob, float* slot_conf, uint8_t* slot_selected,
                                int32_t* n_selected, int32_t* verify_row_offsets,
                                int32_t* verify_src_rows, int32_t* verify_tokens,
                                const zarya_sample_desc* desc, zarya_stream_t stream);

/*
 * Step 6. desc->row_offsets is the verification layout (verify_row_offsets
 * of the draft); n_slots[b] is the number of verified slots (n_selected of
 * the draft, 0 allowed), slot_len[b] = L_b; tokens [total_rows] int32 holds
 * the token of every verification row (verify_tokens of the draft).
 * Outputs (device, written):
 *  token_prob  [total_rows] float        probability of the row's token (0, with
 *                                        ZARYA_DEVERR_TOKEN, for a token outside [0, V))
 *  slot_accept [B, max_slots] int32      accepted prefix of verified slot k (0 past n_slots[b])
 *  accept_len  [B] int32                 accepted prefix of the sequence's verification
 *                                        rows (0 .. n_slots[b] * L_b)
 * Rows outside every sequence are not read or written.
 */
zarya_status zarya_verify_accept(const void* logits, const int32_t* tokens,
                                 const int32_t* n_slots, const int32_t* slot_len,
                                 float* token_prob, int32_t* slot_accept, int32_t* accept_len,
                                 const zarya_sample_desc* desc, zarya_stream_t stream);

/*
 * Steps 3-4 of either mode without the selection: the draw and its
 * probability for every row of the sequences in desc->row_offsets (row r of
 * [row_offsets[0], row_offsets[B])), as defined above (argmax at T = 0,
 * Gumbel-max over the Philox noise at T > 0). In Mode A these are the rows of
 * the positions a step reveals (Sec. 5.1 step 3). n_slots / slot_len and the
 * thresholds of desc are not used.
 *  tokens [total_rows] int32, prob [total_rows] float (written for those rows)
 */
zarya_status zarya_sample_rows(const void* logits, int32_t* tokens, float* prob,
                               const zarya_sample_desc* desc, zarya_stream_t stream);

/* ------------------------------------------------------------------------
 * Mode A mask-budget planning (Sec. 5.1 step 1).
 *
 * For sequence b with n = n_masked[b] masked tokens: with T > 0, exactly T
 * diffusion steps reveal Binomial(n, alpha0) of them, diffusion step s (of T)
 * revealing Binomial(r_s, 1 / (T - s)) of the r_s not yet revealed (the last
 * takes the rest), and the remaining n - n_diff tokens are revealed one per
 * step after them; with T = 0 the noise is ignored: ceil(n / 4) steps of 4
 * (the last takes the remainder); n = 0 gives no step. Each binomial draw is
 * the sum of Bernoulli trials [u_i < p] (p in fp32) with u_i the uniform
 * defined above, from Philox4x32-10 with key (seed low, seed high) and counter
 * (i / 4, b, draw, offset low word), word i % 4; draw 0 is the diffusion
 * total, draw 1 + s diffusion step s.
 *  n_masked [batch] int32 (read; negative sets ZARYA_DEVERR_ROWS)
 *  counts   [batch, max_steps] int32 (written: reveal count of each step, 0 after the plan)
 *  n_steps  [batch] int32 (written; 0 with ZARYA_DEVERR_ROWS when the plan has more than
 *           max_steps steps)
 */
zarya_status zarya_mode_a_budget(const int32_t* n_masked, int32_t batch, int32_t T, float alpha0,
                                 uint64_t seed, uint64_t offset, int32_t max_steps,
                                 int32_t* counts, int32_t* n_steps, zarya_stream_t stream);

/* ------------------------------------------------------------------------
 * Reordering and restoration (Sec. 5.1 steps 2 and 4, Sec. 5.2 steps 1 and 8).
 *
 * Before the first forward pass a sequence is reordered so that every
 * unmasked (visible) token comes before every masked one; after the last
 * step it is restored to the original order. Sequences are the rows of
 * [batch, max_len] arrays: sequence b's tokens are its first lens[b]
 * positions (0 <= lens[b] <= max_len; otherwise ZARYA_DEVERR_ROWS and the
 * sequence is treated as empty). Positions at or past lens[b] are copied
 * through unchanged and get perm -1.
 */

/*
 * perm[b, i] = the original position of reordered position i: the unmasked
 * positions in their order, then the masked positions in their order or,
 * when order_key is given, by ascending (order_key, position) (the token
 * shuffling of Mode A, Table 2). perm doubles as the position ids of the
 * reordered sequence. tokens_out[b, i] = tokens[b, perm[b, i]];
 * n_unmasked[b] = the number of unmasked positions (the prefix length of the
 * reordered sequence).
 *  tokens     [batch, max_len] int32 (read)
 *  is_masked  [batch, max_len] uint8 (read; nonzero = masked)
 *  order_key  [batch, max_len] uint32 (read) or NULL
 *  lens       [batch] int32 (read)
 *  perm, tokens_out [batch, max_len] int32 (written; tokens_out must not
 *             overlap tokens)
 *  n_unmasked [batch] int32 (written)
 */
zarya_status zarya_reorder(const int32_t* tokens, const uint8_t* is_masked,
                           const uint32_t* order_key, const int32_t* lens, int32_t batch,
                           int32_t max_len, int32_t* perm, int32_t* tokens_out,
                           int32_t* n_unmasked, zarya_stream_t stream);

/*
 * tokens_out[b, perm[b, i]] = tokens[b, i] for i < lens[b] (perm as written
 * by zarya_reorder); positions past lens[b] copied through. A perm entry
 * outside [0, lens[b]) sets ZARYA_DEVERR_PERM and is skipped. tokens_out
 * must not overlap tokens.
 */
zarya_status zarya_restore(const int32_t* tokens, const int32_t* perm, const int32_t* lens,
                           int32_t batch, int32_t max_len, int32_t* tokens_out,
                           zarya_stream_t stream);

/*
 * Repetition penalty (Sec. 5.1 step 3 and Table 2: the per-step draws honour
 * temperature, top_p and repetition_penalty; the paper names the parameter,
 * and the reading here is the usual one for a generate() call): in place, for
 * every row g of sequence b (rows desc->row_offsets[b] .. [b + 1] - 1) and
 * every distinct token v among hist_tokens[hist_offsets[b] ..
 * hist_offsets[b + 1] - 1], the logit x = logits[g, v] becomes x * penalty
 * when x < 0 and x / penalty otherwise, computed in float32 (bf16 logits are
 * rounded back to nearest even). A token that occurs several times is
 * penalised once. Run it on the logits before zarya_draft_select,
 * zarya_verify_accept or zarya_sample_rows.
 *  logits       [desc->total_rows, desc->row_stride] of desc->dtype (read and
 *               written; 16-byte aligned); rows of no sequence are untouched
 *  hist_offsets [desc->batch + 1] int32, non-decreasing, last <= n_hist
 *  hist_tokens  [n_hist] int32 (may be NULL when n_hist is 0)
 *  penalty      > 0 and finite (1 changes nothing)
 * desc supplies batch, vocab, dtype, total_rows, row_stride and row_offsets;
 * its other fields are checked as for zarya_draft_select but not used.
 * Device checks: a history range outside [0, n_hist] sets ZARYA_DEVERR_ROWS
 * and leaves that row alone; a token outside [0, vocab) sets
 * ZARYA_DEVERR_TOKEN and is skipped. Vocabularies above 1.6 M tokens return
 * ZARYA_ERR_UNSUPPORTED.
 */
zarya_status zarya_repetition_penalty(void* logits, const int32_t* hist_offsets,
                                      const int32_t* hist_tokens, int32_t n_hist, float penalty,
                                      const zarya_sample_desc* desc, zarya_stream_t stream);

/*
 * top_p (nucleus) truncation (Sec. 5.1 step 3 and Table 2; the paper names
 * the parameter, and the reading here is nucleus sampling): in place, for
 * every row of a sequence (rows desc->row_offsets[0] .. [batch] - 1), with
 * p = softmax(x / T) (softmax(x) when desc->temperature is 0), the logits
 * below x* become -inf, where x* is the largest logit value such that the
 * tokens at or above it hold at least top_p of the row's probability: the
 * smallest set of most probable tokens reaching top_p, with every token tied
 * at its boundary kept. A draw that follows (zarya_draft_select,
 * zarya_verify_accept, zarya_sample_rows with the same temperature) then runs
 * over the nucleus, each token with its usual noise, and reports
 * probabilities renormalised over it. The masses behind the boundary are
 * summed in fixed point (each token's mass to 2^-21 of itself), so the result
 * does not depend on the order of the GPU's additions; it can differ from
 * exact arithmetic only where the mass at a boundary lies within about 1e-6 of
 * top_p.
 *  logits   [desc->total_rows, desc->row_stride] of desc->dtype (read and
 *           written; 16-byte aligned); rows of no sequence are untouched,
 *           and NaN logits are left in place (they carry no mass)
 *  top_p    in (0, 1); top_p >= 1 returns at once (nothing to cut)
 * desc supplies batch, vocab, dtype, total_rows, row_stride, row_offsets and
 * temperature; its other fields are checked as for zarya_draft_select.
 * Returns ZARYA_ERR_INVALID_ARG for top_p <= 0 or NaN, and
 * ZARYA_ERR_UNSUPPORTED for a vocabulary above 520,192 tokens.
 */
zarya_status zarya_top_p(void* logits, float top_p, const zarya_sample_desc* desc,
                         zarya_stream_t stream);

/*
 * Moves `bytes` bytes from src to dst with a kernel instead of a copy engine:
 * a grid of at most 24 CTAs reads and writes 16-byte vectors, reaching host
 * memory through its device mapping. Each of src and dst is device memory or
 * page-locked host memory the device can address (cudaHostAlloc /
 * cudaMallocHost, or cudaHostRegister with the mapped flag; with unified
 * addressing every page-locked allocation is mapped); at least one is device
 * memory. Meant for a step's inputs and outputs: inside a CUDA graph the copy
 * is one more kernel node, with none of the copy-engine hand-over a memcpy
 * node costs next to kernels. Not a step of the paper's method.
 *  src, dst: 16-byte aligned, ranges not overlapping; bytes: any (0 launches
 *            nothing). Ordered on `stream` like any kernel.
 * The device is the stream's (or, while capturing or on the legacy stream,
 * that of the device buffer); device memory must belong to it.
 * Returns ZARYA_ERR_INVALID_ARG (nothing launched) for a NULL or unaligned
 * pointer, memory the device cannot address (another device's memory,
 * pageable host memory), two host buffers, or overlapping ranges.
 */
zarya_status zarya_copy(const void* src, void* dst, size_t bytes, zarya_stream_t stream);

/*
 * Synchronises `stream`, then reads and clears the error word of the device
 * that owns it. Returns ZARYA_OK when it was clear, ZARYA_ERR_DEVICE_FAULT
 * when it was set (*code receives its ZARYA_DEVERR_* value; code may be
 * NULL), ZARYA_ERR_CUDA when the synchronisation itself failed.
 */
zarya_status zarya_check_device_error(zarya_stream_t stream, int32_t* code);

/*
 * Message about the last CUDA runtime/driver failure behind a ZARYA_ERR_CUDA
 * returned on the calling thread ("what failed: CUDA's error string (code)");
 * empty if there was none. Owned by the library; valid until the next call
 * on the same thread.
 */
const char* zarya_last_error(void);

/* Static, human-readable name of a status. */
const char* zarya_status_string(zarya_status status);

/* Library version, major * 10000 + minor * 100 + patch. */
int32_t zarya_version(void);

#ifdef __cplusplus
}
#endif

#endif /* ZARYA_H_ */
