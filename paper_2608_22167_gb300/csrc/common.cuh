// Device-side building blocks shared by the kernels of the paged-attention
// path: inline-PTX wrappers (mbarrier, TMA tensor loads, ldmatrix, mma.sync,
// movmatrix), the swizzled shared-memory addressing that matches the TMA
// 128-byte swizzle, the device status word and the work-plan records that the
// planner kernel writes into the caller's workspace.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace mcpu {

// ----------------------------------------------------------------- geometry
constexpr int kHeadDim = 64;          // D; one key row = 128 bytes of bf16
constexpr int kPage = 16;             // tokens per page
constexpr int kRowBytes = kHeadDim * 2;
constexpr int kTileBytes = kPage * kRowBytes;  // one (page, kv head) block: 2 KiB
constexpr int kMaxSeqs = 2048;        // rows per call handled by the planner
constexpr int kPlanThreads = 1024;
constexpr int kRowsPerPlanThread = kMaxSeqs / kPlanThreads;
constexpr int kMaxGroup = 8;          // largest supported H_q / H_kv
constexpr int kSplitBudget = 4096;    // bound on member-weighted KV splits per call
constexpr int kMinSplitPages = 8;     // shortest split of a decode row, in pages
constexpr int kMinSharedPages = 4;    // shortest prefix worth a cascade pass
constexpr int kAppendRowsMin = 64;    // smallest append tile (query rows = tokens x heads)
constexpr int kAppendTcRows = 256;    // query rows of one tcgen05 append item (two 128-row tiles)

// Status bits, OR-ed into the first word of the workspace. They are sticky
// until the caller resets them.
constexpr int32_t kStatusBadPage = 1;
constexpr int32_t kStatusBadLengths = 2;
constexpr int32_t kStatusTimeout = 4;
constexpr int32_t kStatusPlanOverflow = 8;
constexpr int32_t kStatusPoolExhausted = 16;
constexpr int32_t kStatusUnsupportedRow = 32;  // a row the called variant does not handle (skipped)

// Bounded waits: a wait that has not completed after this many nanoseconds
// of %globaltimer gives up and reports kStatusTimeout.
constexpr uint64_t kWaitTimeoutNs = 200ull * 1000ull * 1000ull;

// ------------------------------------------------------------- plan records
struct DecodeItem {   // one KV split of one decode row (all kv heads)
  int32_t row, token, seq_len, first_key;
  int32_t page_begin, page_end, slot, pad;  // slot < 0: write out/lse directly
};
struct CascadeItem {  // one split of a shared prefix, for a subgroup of rows
  int32_t member_off, n_members, page_begin, page_end;
  int32_t split, first_row, pad0, pad1;
};
struct CascadeMember {
  int32_t row, token, part_off, pad;
};
struct AppendItem {   // one tile of query tokens of one append row
  int32_t row, token_begin, n_tok, seq_len;
  int32_t pos_begin, key_begin, key_end, pad;  // keys [key_begin, key_end)
};
struct MergeRow {
  int32_t token, n_parts, part_off, pad;
};

struct PlanHeader {
  int32_t status;
  int32_t n_decode;      // DecodeItem records (kernel items = n * H_kv)
  int32_t n_cascade;     // CascadeItem records
  int32_t n_append;      // AppendItem records
  int32_t n_merge;       // MergeRow records
  int32_t split_pages;   // chosen split length, for inspection
  int32_t n_parts;       // partial slots in use
  int32_t append_ticket; // dynamic scheduler counters, reset by the planner
  int32_t decode_ticket;
  int32_t cascade_ticket;
  int32_t pad[54];
};
static_assert(sizeof(PlanHeader) == 256, "header is one 256-byte block");

// Byte offsets of every array inside the workspace, derived from the dims.
struct WorkspaceLayout {
  size_t header, decode_items, cascade_items, members, append_items, merge_rows;
  size_t lcp;  // per row: leading physical pages equal to the previous row's (shared-prefix scan)
  size_t o_part, lse_part, total;
  int32_t max_decode, max_cascade, max_append, max_parts;
};

__host__ __device__ inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

__host__ __device__ inline WorkspaceLayout workspace_layout(int32_t num_seqs, int32_t total_q,
                                                            int32_t num_q_heads, int32_t group) {
  WorkspaceLayout w;
  int32_t tile_tok = kAppendRowsMin / group;
  w.max_decode = num_seqs + kSplitBudget + 1;
  w.max_cascade = num_seqs / 2 + kSplitBudget + 1;
  w.max_append = total_q / tile_tok + num_seqs + 1;
  w.max_parts = 2 * num_seqs + kSplitBudget + 1;
  size_t off = 0;
  w.header = off;        off += sizeof(PlanHeader);
  w.decode_items = off;  off = align_up(off + sizeof(DecodeItem) * (size_t)w.max_decode, 256);
  w.cascade_items = off; off = align_up(off + sizeof(CascadeItem) * (size_t)w.max_cascade, 256);
  w.members = off;       off = align_up(off + sizeof(CascadeMember) * (size_t)(num_seqs + 1), 256);
  w.append_items = off;  off = align_up(off + sizeof(AppendItem) * (size_t)w.max_append, 256);
  w.merge_rows = off;    off = align_up(off + sizeof(MergeRow) * (size_t)(num_seqs + 1), 256);
  w.lcp = off;           off = align_up(off + sizeof(int32_t) * (size_t)(num_seqs + 1), 256);
  w.o_part = off;        off = align_up(off + sizeof(float) * (size_t)w.max_parts * num_q_heads * kHeadDim, 256);
  w.lse_part = off;      off = align_up(off + sizeof(float) * (size_t)w.max_parts * num_q_heads, 256);
  w.total = off;
  return w;
}

// Arguments every attention kernel receives (by value).
struct AttnParams {
  const __nv_bfloat16* q;        // [T, Hq, D]
  const int32_t* block_table;    // [B, max_pages]
  const int32_t* seq_lens;       // [B]
  const int32_t* qsl;            // [B + 1]
  __nv_bfloat16* out;            // [T, Hq, D]
  float* lse;                    // [T, Hq]
  uint8_t* ws;                   // workspace base
  WorkspaceLayout lay;
  int32_t num_seqs, total_q, max_pages, num_pages;
  int32_t num_q_heads, num_kv_heads, group;
  int32_t window;                // <= 0: none
  float scale_log2;              // softmax scale * log2(e)
  int32_t total_warps_hint;      // resident warps of the decode kernel, for split sizing
  int32_t forced_split_pages;    // > 0: use this split length
  int32_t cascade_enabled;
  int32_t oob_row;               // y coordinate just past the pool, read as zeros
  int32_t append_tile_tok;       // tokens per append tile (tile rows / group)
  const float* sinks;            // [Hq] sink logits (natural log), or null
  int32_t decode_only;           // 1: rows with L > 1 are reported and skipped (fp8 pools)
  // read only by the self-test form of the append kernel: the role that
  // stalls and the report it writes (mcpu_selftest_append_abort)
  int32_t selftest_stall = -1;
  int64_t* selftest_report = nullptr;
};

// Attention sinks (gpt-oss): q head h has a logit sigma_h that joins the
// softmax normaliser and carries no value. sink_log2 is sigma_h in base-2
// units (-inf without sinks). finish_with_sink normalises an accumulator held
// relative to the base-2 running max m with row sum l, the sink included:
// returns the factor the accumulator is multiplied by and writes the base-2
// log normaliser; m may be -inf (no visible key).
__device__ __forceinline__ float sink_log2(const AttnParams& p, int h) {
  return p.sinks ? p.sinks[h] * 1.4426950408889634f : -INFINITY;
}
__device__ __forceinline__ float finish_with_sink(float m, float l, float s2, float* lse2) {
  const float M = fmaxf(m, s2);
  if (!(M > -INFINITY)) {
    *lse2 = -INFINITY;
    return 0.f;
  }
  const float a = m > -INFINITY ? exp2f(m - M) : 0.f;
  const float lt = l * a + (s2 > -INFINITY ? exp2f(s2 - M) : 0.f);
  *lse2 = M + __log2f(lt);
  return a / lt;
}

__device__ __forceinline__ PlanHeader* header(const AttnParams& p) {
  return reinterpret_cast<PlanHeader*>(p.ws + p.lay.header);
}
__device__ __forceinline__ void raise_status(const AttnParams& p, int32_t bits) {
  atomicOr(&header(p)->status, bits);
}

// -------------------------------------------------------------- PTX helpers
__device__ __forceinline__ uint32_t smem_addr(const void* ptr) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(ptr));
}

__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Programmatic dependent launch. A grid launched with programmatic stream
// serialization may begin while the grid before it on the stream still
// runs: grid_dep_wait() returns once that grid has completed and its memory
// operations are visible (at once when the launch was an ordinary one), and
// grid_dep_launch() lets the next grid of the stream launch before this one
// has ended (a CTA that exits counts as having called it).
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
// The same with a suspend-time hint: the thread may sleep in the
// instruction (woken when the phase completes) for up to hint_ns instead of
// returning at once, so a waiting warp does not take issue slots from the
// warps beside it on its sub-partition.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}
// Bounded wait with sleeping polls: false after kWaitTimeoutNs.
__device__ __forceinline__ bool mbar_wait_sleep(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait_sleep(bar, parity, 10000)) {
    if (global_timer_ns() - t0 > kWaitTimeoutNs) return false;
  }
  return true;
}

// Waits for the phase with the given parity to complete; false after
// kWaitTimeoutNs without completion.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitTimeoutNs) return false;
  }
  return true;
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}

// 2-D tiled TMA load of a box into shared memory, completion signalled on
// the mbarrier as transaction bytes.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int32_t x, int32_t y,
                                            uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void prefetch_tensormap(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                                  uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// D = A(16x16, row) * B(16x8, col) + D, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                               uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// The same with fp16 inputs.
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                              uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Untiled bulk copy global -> shared (16-byte aligned addresses, size a
// multiple of 16), completion signalled on the mbarrier as transaction bytes.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                          uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::
          "r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}

// Transpose of an 8x8 matrix of 16-bit elements held one row-pair per lane.
__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Byte offset of 16-byte chunk `chunk` (0..7) of row `row` in a tile of
// 128-byte rows written by TMA with 128-byte swizzling (tile base 1024-aligned):
// the chunk index is XOR-ed with the row index modulo 8.
__device__ __forceinline__ uint32_t swz128(int row, int chunk) {
  return static_cast<uint32_t>(row * 128 + ((chunk ^ (row & 7)) << 4));
}

__device__ __forceinline__ float fast_exp2(float x) { return exp2f(x); }

// Packed fp32 pairs (two lanes of a 64-bit register): d = a * b + c and d = a + b.
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t pack_f32x2(float lo, float hi) {
  return (uint64_t)__float_as_uint(lo) | ((uint64_t)__float_as_uint(hi) << 32);
}
__device__ __forceinline__ float lo_f32(uint64_t v) { return __uint_as_float((uint32_t)v); }
__device__ __forceinline__ float hi_f32(uint64_t v) { return __uint_as_float((uint32_t)(v >> 32)); }
// max of three floats in one instruction
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// 2^x with the hardware approximation (MUFU.EX2; subnormal results flush to
// zero). Used where the result is rounded to bf16 right after.
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Launch configuration of one kernel, with programmatic stream serialization
// when `programmatic` is set (the kernel then waits with grid_dep_wait()
// before it uses the previous grid's results). Used in place: `cfg.attrs`
// points into the object.
struct LaunchCfg {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  LaunchCfg(dim3 grid, dim3 block, size_t smem, cudaStream_t stream, bool programmatic) {
    cfg = cudaLaunchConfig_t{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = programmatic ? 1 : 0;
  }
  LaunchCfg(const LaunchCfg&) = delete;
  LaunchCfg& operator=(const LaunchCfg&) = delete;
};

}  // namespace mcpu
