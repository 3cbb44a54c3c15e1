/*
 * mcpu.h -- C ABI of the GB300 (sm_103a) paged-attention hot path.
 *
 * The paper (MCP-Universe RL, §3.2) describes a rollout engine that keeps
 * hundreds of multi-turn tool-use trajectories in flight and notes that the
 * run stage is bound by GPU generation. Between tool calls every trajectory
 * either decodes one token or appends a tool-observation chunk, and the n = 8
 * samples of a GRPO task (§4; App. B, Tab. "hparams") share their prompt.
 * This library is that generation step's attention: a ragged batch of rows
 * ("trajectories") whose KV caches live in a paged pool, with
 *
 *   mcpu_kv_append                -- writes the new tokens' K/V into their pages
 *   mcpu_paged_attention_forward  -- causal (optionally sliding-window)
 *                                    softmax attention of every query token
 *                                    over its row's paged keys and values,
 *                                    returning out and the log-sum-exp
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every pointer argument except `dims`/`opts`/`status_bits` and the
 *    `*_host` arguments of mcpu_paged_attention_host is DEVICE memory owned
 *    by the caller; the library never frees or retains it.
 *    Tensors are dense, row-major, with the shapes given below. bf16 data and
 *    the pools must be 16-byte aligned.
 *  - Work is enqueued on `stream` (NULL = the legacy default stream) and the
 *    call returns without synchronising. The forward call allocates nothing:
 *    all scratch lives in the caller's workspace.
 *  - Host-side argument checks return an error code synchronously and launch
 *    nothing. Errors only visible on the device (a page id outside the pool,
 *    L_r > S_r, a wait that timed out) set bits in a status word at the start
 *    of the workspace and the kernels skip or zero-fill the affected reads;
 *    read it with mcpu_read_device_status. Nothing traps.
 *
 * Notation (row r = one trajectory):
 *   B  = num_seqs, T = total_q = query_start_loc[B]
 *   L_r = query_start_loc[r+1] - query_start_loc[r]  (1 for a decode row)
 *   S_r = seq_lens[r]: KV length of row r AFTER this step's append; the row's
 *         query tokens occupy positions S_r - L_r .. S_r - 1.
 *   Query i of row r sits at p = S_r - L_r + i and sees key j iff j <= p and,
 *   when sliding_window W > 0, p - j < W. q head h reads kv head h / (H_q/H_kv).
 *
 * Layouts:
 *   q             [T, H_q, D]          bf16
 *   k_new, v_new  [T, H_kv, D]         bf16  (one row per query token)
 *   k_cache, v_cache [num_pages, H_kv, page_size, D] bf16: the (page, kv head)
 *                 block is page_size * D * 2 contiguous bytes.
 *   block_table   [B, max_pages_per_seq] int32: logical page -> physical page.
 *                 Entries no query can see may hold anything (e.g. -1).
 *                 Slots of a page that no query of the call can see (never
 *                 written yet, or before a window) may hold anything, NaN
 *                 and Inf included: the kernels give them no weight and zero
 *                 their V rows before the weighted sum.
 *   seq_lens      [B] int32;  query_start_loc [B + 1] int32 (prefix sums, [0] = 0)
 *   out           [T, H_q, D] bf16;  lse [T, H_q] float (natural log of the
 *                 softmax normaliser sum_j exp(scale * q.k_j); -inf if empty)
 *
 * Supported now: D = 64, page_size = 16, H_q / H_kv in {1, 2, 4, 8},
 * num_seqs <= 2048. Anything else returns MCPU_ERR_UNSUPPORTED.
 */
#ifndef MCPU_H
#define MCPU_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t (a CUstream_st pointer). */
typedef struct CUstream_st* mcpu_stream_t;

typedef enum mcpu_status {
  MCPU_OK = 0,
  MCPU_ERR_INVALID_ARG = 1,          /* null/misaligned pointer, inconsistent dims */
  MCPU_ERR_UNSUPPORTED = 2,          /* valid but not implemented (D, page size, ratio) */
  MCPU_ERR_WORKSPACE_TOO_SMALL = 3,  /* workspace_bytes < mcpu_workspace_size(dims) */
  MCPU_ERR_CUDA = 4,                 /* a CUDA runtime call failed (launch, attributes) */
  MCPU_ERR_BAD_PAGE = 5,             /* device: a needed block-table entry is outside the pool */
  MCPU_ERR_BAD_LENGTHS = 6,          /* device: L_r > S_r, L_r < 0, S_r beyond the table, or
                                        query_start_loc[0] != 0 / [B] != total_q */
  MCPU_ERR_TIMEOUT = 7,              /* device: a bounded wait gave up */
  MCPU_ERR_INTERNAL = 8,             /* device: work plan overflowed its bound */
  MCPU_ERR_POOL_EXHAUSTED = 9,       /* device: the free-page stack ran empty */
  MCPU_ERR_UNSUPPORTED_ROW = 10      /* device: a row the called variant does not handle was
                                        skipped (an append row given to the fp8 forward) */
} mcpu_status;

typedef struct mcpu_dims {
  int32_t num_seqs;           /* B */
  int32_t total_q;            /* T = query_start_loc[B] */
  int32_t max_pages_per_seq;  /* columns of block_table */
  int32_t num_pages;          /* physical pages in each of k_cache / v_cache */
  int32_t num_q_heads;        /* H_q */
  int32_t num_kv_heads;       /* H_kv */
  int32_t head_dim;           /* D (64) */
  int32_t page_size;          /* tokens per page (16) */
} mcpu_dims;

/* Optional knobs of the forward pass; pass NULL for the defaults. */
#define MCPU_FLAG_NO_CASCADE 0x1u       /* never run the shared-prefix (cascade) pass */
#define MCPU_FLAG_MMA_SYNC_APPEND 0x2u  /* append chunks on the mma.sync kernel instead of tcgen05 */
#define MCPU_FLAG_SERIAL 0x4u           /* run every kernel on `stream` (no side stream) */
#define MCPU_FLAG_HOST_OUT_DIRECT 0x8u  /* host-buffer calls: kernels write out/lse straight into page-locked host memory;
                                           forward calls: out/lse are page-locked host memory, written in whole sectors */
typedef struct mcpu_options {
  uint32_t flags;             /* MCPU_FLAG_* */
  int32_t split_pages;        /* > 0: KV split length of decode rows, in pages (0 = auto) */
  /* Optional timing hook: if non-NULL, MCPU_NUM_PHASE_EVENTS cudaEvent_t
   * handles (created by the caller) that the call records: [0] before the
   * planner, [1] after it, [2] after split-KV decode, [3] after the cascade
   * pass, [4] after the append-chunk kernel, [5] after the merge. By default
   * decode and cascade run, in that order, on the library's side stream
   * concurrently with the append kernel on `stream`: then [2] and [3] are
   * recorded on the side stream and the append kernel spans [1]..[4].
   * Under stream capture they become event-record nodes of the graph, so
   * every replay records them. */
  void* const* phase_events;
  /* Optional attention sinks (gpt-oss; not in the paper): device pointer to
   * H_q floats, the sink logit sigma_h of each q head in natural-log units,
   * or NULL. A sink joins the softmax normaliser and carries no value:
   * out = sum_j e^{s_j} V_j / (sum_j e^{s_j} + e^{sigma_h}) and lse is the
   * log of that normaliser. 4-byte aligned; read by the kernels only. */
  const float* sinks;
} mcpu_options;
#define MCPU_NUM_PHASE_EVENTS 6

/* Bytes of workspace mcpu_paged_attention_forward needs for these dims
 * (depends on num_seqs, total_q and the head counts only). 0 if dims are
 * invalid. The first 4 bytes are the device status word: zero the workspace
 * once before first use (or call mcpu_reset_device_status). */
size_t mcpu_workspace_size(const mcpu_dims* dims);

/*
 * KV append (the new tokens of every row enter the cache): the step between
 * two generations of a trajectory in which the tool observation's tokens (an
 * append row) or the token just generated (a decode row) join its context
 * (paper §3.2, the run stage's alternation of generation and tool calls).
 * For each row r and i < L_r, copies k_new[query_start_loc[r] + i] (all kv
 * heads) bit for bit to k_cache[block_table[r][pos / page]][h][pos % page]
 * with pos = S_r - L_r + i; likewise v_new into v_cache. Decode rows append
 * their one token; append rows their whole chunk. Nothing else is written.
 * `status_word` (device int32, may be the workspace start) receives
 * device-side error bits; a row with an invalid page or length is skipped.
 */
mcpu_status mcpu_kv_append(const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                           const int32_t* block_table, const int32_t* seq_lens,
                           const int32_t* query_start_loc, const mcpu_dims* dims,
                           int32_t* status_word, mcpu_stream_t stream);

/*
 * Paged attention forward over a mixed batch of decode rows (L_r = 1) and
 * append rows (L_r > 1, causal within the chunk), with an optional sliding
 * window (W <= 0: full context). This is the attention of the generation
 * that bounds the run stage (paper §3.2; again §4.2): hundreds of
 * trajectories in flight, each either generating one token or taking in a
 * tool observation, the n = 8 samples of a GRPO task sharing their prompt
 * (§4; App. B, Tab. "hparams"), sequences up to 128k tokens. Rows with L_r = 0 produce nothing.
 * softmax_scale (> 0, finite) multiplies q.k (1/sqrt(D) for gpt-oss). Rows that are
 * adjacent in the batch and whose block tables start with the same physical
 * pages (a GRPO group's shared prompt) are detected on the device and their
 * common full pages are read once for the whole group (full-context calls
 * only). Long decode rows are split over SMs and merged by log-sum-exp.
 * Results do not depend on the split or cascade choices beyond rounding.
 * The memory-bound decode kernels run concurrently with the tensor-core
 * append kernel: the call forks them, the cascade pass and the merge onto a
 * library-owned, low-priority stream of the current device after the
 * planner and joins back at the end, with CUDA events. Pass
 * MCPU_FLAG_SERIAL to keep every kernel on `stream`. Set
 * MCPU_FLAG_HOST_OUT_DIRECT when out and lse are page-locked host memory
 * the device can address: the append kernel then writes out in 32-byte
 * pieces (whole sectors, if out is 32-byte aligned), which the host link
 * takes far better than 16-byte halves of sectors (device memory gives the
 * same results that way). The call is capturable in a CUDA graph (with mcpu_kv_append
 * before it): it allocates nothing, synchronises nothing, and its work plan
 * is rebuilt on the device at every replay, so a replayed graph follows
 * changed seq_lens / block_table / query_start_loc contents as long as the
 * dims (and hence the pointers' extents) stay the same. The first call on a
 * device sets kernel attributes and creates the side stream; make it before
 * any capture.
 */
mcpu_status mcpu_paged_attention_forward(const void* q, const void* k_cache, const void* v_cache,
                                         const int32_t* block_table, const int32_t* seq_lens,
                                         const int32_t* query_start_loc, int32_t sliding_window,
                                         float softmax_scale, const mcpu_dims* dims, void* out,
                                         float* lse, void* workspace, size_t workspace_bytes,
                                         const mcpu_options* opts, mcpu_stream_t stream);

/*
 * Paged attention forward for callers that cannot allocate device memory
 * (an engine that reserves all GPU memory up front, code running under CUDA
 * graph stream capture, a host that only receives device pointers). It has
 * no counterpart in the paper: it is a deployment variant of
 * mcpu_paged_attention_forward that takes no workspace. Its scratch (status
 * word and work plan) lives in a 4 MiB array in the library's own device
 * memory, held by every GPU that loads the library until the process exits.
 *
 * Same arguments and results as mcpu_paged_attention_forward (up to
 * rounding), except:
 *  - no workspace and no options: decode rows are not split across SMs and
 *    the shared-prefix pass is off, so long decode rows run slower;
 *  - total_q <= 262144 (num_seqs <= 2048 as for the other entry point);
 *    larger batches return MCPU_ERR_WORKSPACE_TOO_SMALL without launching;
 *  - `status_word` (device int32, may be NULL) receives this call's device
 *    status bits (same meaning as the workspace status word), copied on
 *    `stream` after the kernels.
 * Every call on a device shares the one scratch array, which keeps the last
 * call's contents (the call clears the status word itself): calls that
 * overlap on the GPU (different streams, no ordering between them) race.
 * The first call on a device looks up the array's device address and sets
 * kernel attributes; make that first call before any stream capture.
 */
mcpu_status mcpu_paged_attention_forward_noalloc(const void* q, const void* k_cache, const void* v_cache,
                                                 const int32_t* block_table, const int32_t* seq_lens,
                                                 const int32_t* query_start_loc, int32_t sliding_window,
                                                 float softmax_scale, const mcpu_dims* dims, void* out,
                                                 float* lse, int32_t* status_word, mcpu_stream_t stream);

/*
 * KV append with the rotary position embedding fused in (the rotation gpt-oss
 * applies to q and k before attention; the paper does not describe the
 * model's layers). For each query token t of row r at position
 * p = S_r - L_r + i: q[t] (all H_q heads) is rotated in place, and k_new[t]
 * rotated, v_new[t] as is, are written to (block_table[r][p / 16], p % 16)
 * exactly as mcpu_kv_append writes them (k_new itself is not modified).
 * Rotation of a 64-dim row x by table row p, for i < 32:
 *   y_i = x_i cos_i - x_{i+32} sin_i,  y_{i+32} = x_{i+32} cos_i + x_i sin_i,
 * cos_i = cos_sin[p * 64 + i], sin_i = cos_sin[p * 64 + 32 + i] (device
 * float, max_position rows; the caller builds it for its model), computed in
 * fp32 and rounded once to bf16. Tokens at p >= max_position, or with
 * inconsistent lengths, set MCPU_ERR_BAD_LENGTHS in status_word and are left
 * untouched; a bad page skips that token's K/V write (MCPU_ERR_BAD_PAGE).
 */
mcpu_status mcpu_rope_kv_append(void* q, const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                                const int32_t* block_table, const int32_t* seq_lens,
                                const int32_t* query_start_loc, const float* cos_sin, int32_t max_position,
                                const mcpu_dims* dims, int32_t* status_word, mcpu_stream_t stream);

/*
 * Grows block tables in place on the device (no host round trip): every
 * logical page j < ceil(S_r / 16) of row r whose entry block_table[r][j] is
 * negative receives a page popped from the stack free_pages[0 .. *free_count)
 * (device int32; the top is free_pages[*free_count - 1]); *free_count is
 * decremented accordingly. Entries already set (shared prompt pages, pages of
 * earlier steps) are not touched. Which row gets which popped page is not
 * specified. If the stack runs empty the remaining entries stay negative and
 * MCPU_ERR_POOL_EXHAUSTED is raised in status_word. Uses dims->num_seqs and
 * dims->max_pages_per_seq only. Not a part of the paper's method: the engine
 * bookkeeping either side of the attention call.
 */
mcpu_status mcpu_grow_block_tables(int32_t* block_table, const int32_t* seq_lens, const mcpu_dims* dims,
                                   const int32_t* free_pages, int32_t* free_count, int32_t* status_word,
                                   mcpu_stream_t stream);

/*
 * fp8 KV pages (a storage variant for the memory-bound decode; not in the
 * paper, which keeps K/V in bf16). Each (token, kv head) row x of D = 64
 * values is stored as 64 e4m3 codes (OCP "e4m3fn": bias 7, largest 448,
 * subnormals down to 2^-9, no infinities) and one float scale, computed in
 * float arithmetic as a = max_i |x_i|, scale = a / 448,
 * code_i = e4m3(x_i * (448 / a)) rounded to nearest-even and saturated to
 * +-448 (an all-zero row stores zero codes and scale 0). Attention reads
 * K[j][d] = value(code) * scale. One scale per row rather than per page, so
 * that a page can fill one token at a time without requantizing.
 *
 * Layout: one pool `kv8` of num_pages * H_kv blocks of 2176 bytes, block
 * (page, h) at byte offset (page * H_kv + h) * 2176 (16-byte aligned base):
 *   bytes    0..1023  K codes, uint8 [16 slots][D] (row-major)
 *   bytes 1024..2047  V codes in the decode kernel's MMA-fragment order: for
 *                     half e in {0, 1}, lane l = 4 r + c (r in 0..7, c in
 *                     0..3), j in 0..3 and i in 0..3, byte
 *                     1024 + 512 e + 16 l + 4 j + i holds dim
 *                     16 (2 e + j / 2) + 8 (j % 2) + r of slot 4 c + i
 *   bytes 2048..2175  scales, float: for r in 0..7, the 16 bytes at
 *                     2048 + 16 r hold the K scales of slots a and a + 2,
 *                     then the V scales of slots a and a + 2, where
 *                     a = 4 (r / 2) + r % 2
 * so that one copy brings a page's K, V and scales (a 16-token page takes
 * 2176 bytes per kv head instead of 4096 in bf16) and every operand of a
 * lane is one 16-byte shared-memory load. Slots that no row has written may
 * hold anything: the kernels mask them.
 *
 * mcpu_kv_append_fp8: as mcpu_kv_append (same placement, lengths and error
 * bits), quantizing each new K and V row as above; k_new, v_new stay bf16.
 */
mcpu_status mcpu_kv_append_fp8(const void* k_new, const void* v_new, void* kv8, const int32_t* block_table,
                               const int32_t* seq_lens, const int32_t* query_start_loc, const mcpu_dims* dims,
                               int32_t* status_word, mcpu_stream_t stream);

/*
 * mcpu_paged_attention_forward over fp8 pages, for decode rows (L_r = 1 or
 * 0): same arguments, results and options as mcpu_paged_attention_forward
 * (split-KV, cascade pass over shared prompt pages, sliding window, sinks,
 * phase events, graph capture), with the two bf16 pools replaced by kv8.
 * dims->num_pages counts pages of kv8. The products run on the fp16 tensor
 * cores: codes are converted exactly to fp16; q enters as fp16 times a power
 * of two per query vector (exact for every bf16 entry above 2^-28 of the
 * vector's largest); the softmax weights times the V scales enter as fp16
 * (about 2^-11 relative); accumulation in fp32.
 * A batch with total_q > num_seqs (some row appends) returns
 * MCPU_ERR_UNSUPPORTED without launching; an append row found on the device
 * is skipped and reported as MCPU_ERR_UNSUPPORTED_ROW. MCPU_FLAG_MMA_SYNC_APPEND
 * is not accepted; every kernel runs on `stream`.
 */
mcpu_status mcpu_paged_attention_forward_fp8(const void* q, const void* kv8, const int32_t* block_table,
                                             const int32_t* seq_lens, const int32_t* query_start_loc,
                                             int32_t sliding_window, float softmax_scale, const mcpu_dims* dims,
                                             void* out, float* lse, void* workspace, size_t workspace_bytes,
                                             const mcpu_options* opts, mcpu_stream_t stream);

/*
 * Calls with host buffers (a deployment variant with no counterpart in the
 * paper, whose engine keeps q, K and V on the GPU): one layer's per-token
 * inputs and outputs live in host memory and the library moves them, with
 * the copies overlapped with the attention itself.
 *
 * mcpu_host_stage_create allocates, on the current device, `slots` (2 to
 * MCPU_MAX_HOST_SLOTS) staging slots of device memory (each holds one
 * call's q, k_new, v_new, out, lse and row metadata for up to max_tokens
 * query tokens and max_rows rows with the given head counts; about
 * max_tokens * (4 H_q + 2 H_kv) * 64 bytes each) and two copy streams.
 * Calls take the slots in turn, so the inputs of the next slots - 1 calls
 * can be copied in while one computes (more slots absorb layers whose
 * copies outlast their compute). Returns MCPU_ERR_CUDA if an allocation
 * fails. mcpu_host_stage_destroy frees the stage (NULL is ignored).
 *
 * mcpu_paged_attention_host: mcpu_kv_append followed by
 * mcpu_paged_attention_forward (same arguments, rules and results) with
 *   q_host [T, H_q, D], k_new_host / v_new_host [T, H_kv, D] bf16,
 *   seq_lens_host [B], query_start_loc_host [B + 1] int32: HOST memory;
 *   out_host [T, H_q, D] bf16, lse_host [T, H_q] float: HOST memory;
 *   k_cache, v_cache, block_table, workspace: device memory as before.
 * The rows are cut into `slices` contiguous row ranges of about equal token
 * counts (mcpu_host_slice_rows; at most MCPU_MAX_HOST_SLICES; 0 = two
 * slices from 64 MiB moved, else one; a single row is never cut). Slice s's inputs are copied in on the
 * stage's input stream while slice s - 1 computes, and its outputs are
 * copied out on the output stream while slice s + 1 computes; the compute
 * runs on `stream`, ordered after the work already there.
 * With MCPU_FLAG_HOST_OUT_DIRECT in opts, and out_host and lse_host in
 * page-locked memory the device can address, the kernels write the outputs
 * there themselves as they finish them, over the host link, and nothing is
 * copied back (slices = 0 then means one slice). That suits the call whose
 * outputs are wanted right after it (nothing is left to copy once its last
 * kernel ends); a call followed by more work does better with the copies,
 * which run beside that work, and with slices = 1 (its output copy already
 * overlaps the next call, and each slice adds its own planner and kernel
 * tails). Without the flag, or for other host memory,
 * the outputs are staged and copied. Shared-prefix
 * detection only sees rows within one slice. query_start_loc_host is read
 * on the host during the call; the other host buffers are read or written
 * asynchronously: page-locked memory gives full copy speed, and every host
 * buffer must stay valid, and the inputs unchanged, until the outputs are
 * complete. The outputs of a call are complete once mcpu_host_stage_sync
 * has returned, or, on the device, after a later mcpu_host_stage_wait on
 * `stream`. A stage serves one calling thread at a time. An error after the
 * call has begun enqueuing leaves the stage usable (its later calls and
 * mcpu_host_stage_sync wait for what was enqueued); the outputs are then
 * undefined. mcpu_host_stage_destroy waits for every call's work. Errors: the
 * checks of the two wrapped calls, plus
 * MCPU_ERR_INVALID_ARG when the call exceeds the stage's capacity or head
 * counts, or the current device is not the stage's.
 */
#define MCPU_MAX_HOST_SLICES 8
#define MCPU_MAX_HOST_SLOTS 4
typedef struct mcpu_host_stage mcpu_host_stage;
mcpu_status mcpu_host_stage_create(int32_t max_tokens, int32_t max_rows, int32_t num_q_heads, int32_t num_kv_heads,
                                   int32_t slots, mcpu_host_stage** stage);
mcpu_status mcpu_host_stage_destroy(mcpu_host_stage* stage);
mcpu_status mcpu_paged_attention_host(mcpu_host_stage* stage, const void* q_host, const void* k_new_host,
                                      const void* v_new_host, void* k_cache, void* v_cache,
                                      const int32_t* block_table, const int32_t* seq_lens_host,
                                      const int32_t* query_start_loc_host, int32_t sliding_window,
                                      float softmax_scale, const mcpu_dims* dims, void* out_host, float* lse_host,
                                      void* workspace, size_t workspace_bytes, const mcpu_options* opts,
                                      int32_t slices, mcpu_stream_t stream);
/* mcpu_paged_attention_host over fp8 pages: mcpu_kv_append_fp8 followed by
 * mcpu_paged_attention_forward_fp8 (decode rows; same rules and results)
 * per slice, with the same host buffers, slicing, copies and errors. */
mcpu_status mcpu_paged_attention_host_fp8(mcpu_host_stage* stage, const void* q_host, const void* k_new_host,
                                          const void* v_new_host, void* kv8, const int32_t* block_table,
                                          const int32_t* seq_lens_host, const int32_t* query_start_loc_host,
                                          int32_t sliding_window, float softmax_scale, const mcpu_dims* dims,
                                          void* out_host, float* lse_host, void* workspace, size_t workspace_bytes,
                                          const mcpu_options* opts, int32_t slices, mcpu_stream_t stream);
/* The row ranges mcpu_paged_attention_host uses for `slices` > 0 slices:
 * writes row_begin[0 .. n] (row_begin[0] = 0, row_begin[n] = num_seqs,
 * strictly increasing) and returns the number n of non-empty slices (0 for
 * no rows or invalid arguments). Boundary k is the row whose first token is
 * nearest to k / slices of the total (query_start_loc_host [B + 1], host
 * memory), after the previous boundary; a slice without tokens is dropped.
 * row_begin needs room for slices + 1 entries. Host only. */
int32_t mcpu_host_slice_rows(const int32_t* query_start_loc_host, int32_t num_seqs, int32_t slices,
                             int32_t* row_begin);
/* Makes `stream` wait (on the device) for every output copy the stage has
 * enqueued so far. */
mcpu_status mcpu_host_stage_wait(mcpu_host_stage* stage, mcpu_stream_t stream);
/* Blocks the calling thread until every output copy the stage has enqueued
 * so far is complete. */
mcpu_status mcpu_host_stage_sync(mcpu_host_stage* stage);

/* Synchronises `stream`, reads the workspace status word and maps it to the
 * most severe mcpu_status (MCPU_OK if clear). The raw bits go to
 * *status_bits if non-NULL. The word is not cleared. */
mcpu_status mcpu_read_device_status(const void* workspace, mcpu_stream_t stream, int32_t* status_bits);

/* Enqueues a clear of the workspace status word on `stream`. */
mcpu_status mcpu_reset_device_status(void* workspace, mcpu_stream_t stream);

/* Self-check of the append kernel's abort path (no counterpart in the paper:
 * it exercises, on a GPU and without a fault or a hang, what the tcgen05
 * append kernel does when one of its waits runs out). Runs the planner and
 * then the self-test form of that kernel as ONE CTA over the batch given
 * (same arguments and rules as mcpu_paged_attention_forward; no window, no
 * options; the batch needs an append row whose first work item spans at
 * least two 128-key blocks). In that form one role, chosen by stall_role,
 * stops at the second key block of its first item and waits, for half the
 * library's wait limit, on a barrier nothing completes:
 *   0  the softmax warps of the first query tile,
 *   1  the TMA producer warp,
 *   2  the MMA issuer of the first query tile.
 * It then raises the CTA's abort flag with its own mark (2); every other
 * role, waiting with the full limit, must leave its wait on seeing the flag
 * (a role whose own wait ran out would overwrite the mark with 1, half a
 * limit later), the MMA issuers wait for their MMAs in flight and the
 * producer for its copies in flight, and TMEM is freed. Outputs of the rows
 * are undefined afterwards; the workspace status word gets the timeout bit.
 *   report  device memory, int64_t[16], 8-byte aligned, cleared and written:
 *           [0] the abort flag at the end (2 when only the stalled role ran
 *               out of its wait); [1 + w] nanoseconds from kernel start to
 *               the moment warp w (0..10) left its role; [12] the stalled
 *               wait in ns; [13] the library's wait limit in ns; [14] 1 once
 *               TMEM was freed; [15] unused.
 * Returns MCPU_ERR_INVALID_ARG for a bad role, null or misaligned pointers
 * or an empty batch; otherwise the forward call's errors (asynchronous). */
mcpu_status mcpu_selftest_append_abort(const void* q, const void* k_cache, const void* v_cache,
                                       const int32_t* block_table, const int32_t* seq_lens,
                                       const int32_t* query_start_loc, float softmax_scale, const mcpu_dims* dims,
                                       void* out, float* lse, void* workspace, size_t workspace_bytes,
                                       int32_t stall_role, int64_t* report, mcpu_stream_t stream);

/* Self-check of the device-side timeout path (no counterpart in the paper:
 * it exists so that the path can be exercised on a GPU without a fault or a
 * hang). Every wait in the kernels above is bounded by the library's wait
 * limit (200 ms of the GPU's global timer); when one runs out, the kernel
 * sets the timeout bit of the status word and returns, and
 * mcpu_read_device_status reports MCPU_ERR_TIMEOUT. Inputs cannot cause
 * that, so this call enqueues one small kernel (one CTA) on `stream` in
 * which a warp waits, with the same bounded wait as the decode kernels, on
 * a shared-memory barrier that nothing ever completes, and a second warp on
 * one that does complete. It runs for about the wait limit.
 *   workspace  device memory; only its first 4 bytes (the status word) are
 *              touched: the timeout bit is OR-ed in if the wait gave up.
 *   report     device memory, int64_t[4], 8-byte aligned, written:
 *              [0] 1 if the completing wait returned success, else 0;
 *              [1] 1 if the never-completing wait returned success (a
 *                  failure of the check), else 0;
 *              [2] nanoseconds that wait took; [3] the wait limit in ns.
 * Returns MCPU_ERR_INVALID_ARG for null or misaligned pointers and
 * MCPU_ERR_CUDA if the launch fails; otherwise MCPU_OK (asynchronous). */
mcpu_status mcpu_selftest_wait_timeout(void* workspace, int64_t* report, mcpu_stream_t stream);

/* Static, human-readable name of a status code. */
const char* mcpu_status_string(mcpu_status status);

/* The cudaError_t (as an integer) of the most recent CUDA call that failed
 * inside an entry point of this library (mcpu_kv_append,
 * mcpu_paged_attention_forward, mcpu_paged_attention_forward_noalloc and the
 * others) on the calling thread, i.e. the cause behind its last
 * MCPU_ERR_CUDA; 0 if none has failed. Not cleared by later successful
 * calls. */
int32_t mcpu_last_cuda_error(void);

/* Version of this ABI (bumped on any signature change or addition). */
int32_t mcpu_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* MCPU_H */
