// C ABI of the paged-attention path (declared in include/mcpu.h): host-side
// argument checks, per-device one-time setup (kernel attributes, occupancy),
// TMA descriptors of the two KV pools, and the launch sequence
//   prefix scan -> planner -> append-chunk kernel, and beside it on a side
//   stream: split-KV decode -> cascade pass -> LSE merge
// forked from and joined back into the caller's stream. Nothing here allocates device memory.
#include <cudaTypedefs.h>

#include <mutex>

#include "../../include/mcpu.h"
#include "api_internal.h"
#include "common.cuh"

namespace mcpu {
cudaError_t launch_plan(const AttnParams& p, cudaStream_t stream, bool programmatic);
cudaError_t prepare_plan_kernel();
cudaError_t launch_decode(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttnParams& p, int grid,
                          bool cascade, cudaStream_t stream, bool programmatic);
cudaError_t prepare_decode_kernels(int* bpsm_decode, int* bpsm_cascade);
cudaError_t launch_append(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttnParams& p, int grid,
                          cudaStream_t stream);
cudaError_t prepare_append_kernel(int* bpsm);
cudaError_t launch_append_tc(const CUtensorMap& kmap, const CUtensorMap& vmap, const CUtensorMap& qmap,
                             const AttnParams& p, int grid, bool out_host, cudaStream_t stream);
cudaError_t launch_append_tc_selftest(const CUtensorMap& kmap, const CUtensorMap& vmap, const CUtensorMap& qmap,
                                      const AttnParams& p, cudaStream_t stream);
cudaError_t prepare_append_tc_kernel(int* bpsm);
cudaError_t launch_merge(const AttnParams& p, int grid, cudaStream_t stream, bool programmatic);
cudaError_t prepare_merge_kernel();
cudaError_t prepare_kv_append_kernel();
cudaError_t launch_rope_append(void* q, const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                               const int32_t* block_table, const int32_t* seq_lens, const int32_t* qsl,
                               const float* cos_sin, int32_t max_position, int32_t* status, int32_t num_seqs,
                               int32_t total_q, int32_t max_pages, int32_t num_pages, int32_t num_q_heads,
                               int32_t num_kv_heads, cudaStream_t stream);
cudaError_t launch_grow_tables(int32_t* block_table, const int32_t* seq_lens, int32_t num_seqs, int32_t max_pages,
                               const int32_t* free_pages, int32_t* free_count, int32_t* status,
                               cudaStream_t stream);
cudaError_t launch_kv_append(const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                             const int32_t* block_table, const int32_t* seq_lens, const int32_t* qsl,
                             int32_t* status, int32_t num_seqs, int32_t total_q, int32_t max_pages,
                             int32_t num_pages, int32_t num_kv_heads, cudaStream_t stream);
cudaError_t launch_kv_append_fp8(const void* k_new, const void* v_new, void* kv8, const int32_t* block_table,
                                 const int32_t* seq_lens, const int32_t* qsl, int32_t* status, int32_t num_seqs,
                                 int32_t total_q, int32_t max_pages, int32_t num_pages, int32_t num_kv_heads,
                                 cudaStream_t stream);
cudaError_t launch_decode_fp8(const void* kv8, const AttnParams& p, int grid, bool cascade, cudaStream_t stream,
                              bool programmatic);
cudaError_t prepare_fp8_kernels(int* bpsm_decode, int* bpsm_cascade);
}  // namespace mcpu

namespace {

using namespace mcpu;

constexpr int kMaxDevices = 64;

struct DeviceState {
  bool ready = false;
  int sms = 0;
  int bpsm_decode = 0, bpsm_cascade = 0, bpsm_append = 0, bpsm_append_tc = 0;
  int bpsm_fp8 = 0, bpsm_fp8_cascade = 0;
  // side stream for the memory-bound decode kernels, and the fork/join events
  cudaStream_t side = nullptr;
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
  std::mutex fork_mu;  // one fork/join sequence at a time per device
};

std::mutex g_mu;
DeviceState g_dev[kMaxDevices];

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

mcpu_status device_state(DeviceState** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= kMaxDevices) return MCPU_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceState& st = g_dev[dev];
  if (!st.ready) {
    if (!g_encode) {
      void* fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
              cudaSuccess ||
          q != cudaDriverEntryPointSuccess || fn == nullptr)
        return MCPU_ERR_CUDA;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    if ((e = cudaDeviceGetAttribute(&st.sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_plan_kernel()) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_decode_kernels(&st.bpsm_decode, &st.bpsm_cascade)) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_append_kernel(&st.bpsm_append)) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_append_tc_kernel(&st.bpsm_append_tc)) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_merge_kernel()) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_kv_append_kernel()) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_fp8_kernels(&st.bpsm_fp8, &st.bpsm_fp8_cascade)) != cudaSuccess) return cuda_fail(e);
    if (st.bpsm_decode < 1 || st.bpsm_cascade < 1 || st.bpsm_append < 1 || st.bpsm_append_tc < 1 ||
        st.bpsm_fp8 < 1 || st.bpsm_fp8_cascade < 1)
      return MCPU_ERR_CUDA;
    int lo_prio = 0, hi_prio = 0;
    if ((e = cudaDeviceGetStreamPriorityRange(&lo_prio, &hi_prio)) != cudaSuccess) return cuda_fail(e);
    if ((e = cudaStreamCreateWithPriority(&st.side, cudaStreamNonBlocking, lo_prio)) != cudaSuccess) return cuda_fail(e);
    if ((e = cudaEventCreateWithFlags(&st.ev_fork, cudaEventDisableTiming)) != cudaSuccess) return cuda_fail(e);
    if ((e = cudaEventCreateWithFlags(&st.ev_join, cudaEventDisableTiming)) != cudaSuccess) return cuda_fail(e);
    st.ready = true;
  }
  *out = &st;
  return MCPU_OK;
}

// 2-D view of a pool: rows of D = 64 bf16 (128 bytes), num_pages*H_kv*16 rows;
// boxes of one (page, kv head) block = 16 rows, 128-byte swizzle.
bool encode_pool(CUtensorMap* map, const void* pool, int64_t rows) {
  cuuint64_t dims[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)kRowBytes};
  cuuint32_t box[2] = {(cuuint32_t)kHeadDim, (cuuint32_t)kPage};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(pool), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 3-D view of q [T, H_q, D]: boxes of (256 / g) tokens x the g heads of one kv
// head x 64 dims, i.e. the two 128-row query tiles of an append item, 128-byte
// swizzle.
bool encode_query(CUtensorMap* map, const void* q, int32_t total_q, int32_t num_q_heads, int32_t group) {
  cuuint64_t dims[3] = {(cuuint64_t)kHeadDim, (cuuint64_t)num_q_heads, (cuuint64_t)total_q};
  cuuint64_t strides[2] = {(cuuint64_t)kRowBytes, (cuuint64_t)kRowBytes * num_q_heads};
  cuuint32_t box[3] = {(cuuint32_t)kHeadDim, (cuuint32_t)group, (cuuint32_t)(kAppendTcRows / group)};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(q), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

namespace mcpu {

// most recent failing CUDA call of this thread's entry-point calls
thread_local int32_t t_last_cuda_error = 0;

mcpu_status cuda_fail(cudaError_t e) {
  t_last_cuda_error = (int32_t)e;
  return MCPU_ERR_CUDA;
}

mcpu_status check_dims(const mcpu_dims* d) {
  if (!d) return MCPU_ERR_INVALID_ARG;
  if (d->num_seqs < 0 || d->total_q < 0 || d->max_pages_per_seq < 0 || d->num_pages < 0 || d->num_q_heads <= 0 ||
      d->num_kv_heads <= 0 || d->head_dim <= 0 || d->page_size <= 0)
    return MCPU_ERR_INVALID_ARG;
  if (d->num_q_heads % d->num_kv_heads != 0) return MCPU_ERR_INVALID_ARG;
  if (d->head_dim != kHeadDim || d->page_size != kPage) return MCPU_ERR_UNSUPPORTED;
  const int g = d->num_q_heads / d->num_kv_heads;
  if (g != 1 && g != 2 && g != 4 && g != 8) return MCPU_ERR_UNSUPPORTED;
  if (d->num_seqs > kMaxSeqs) return MCPU_ERR_UNSUPPORTED;
  // pool rows must stay addressable by 32-bit TMA coordinates
  if ((int64_t)d->num_pages * d->num_kv_heads * kPage >= (int64_t)0x7fff0000) return MCPU_ERR_UNSUPPORTED;
  if ((int64_t)d->max_pages_per_seq * kPage >= (int64_t)0x7fff0000) return MCPU_ERR_UNSUPPORTED;
  return MCPU_OK;
}

mcpu_status from_cuda(cudaError_t e) { return e == cudaSuccess ? MCPU_OK : cuda_fail(e); }

}  // namespace mcpu

extern "C" {

int32_t mcpu_abi_version(void) { return 7; }

int32_t mcpu_last_cuda_error(void) { return mcpu::t_last_cuda_error; }

const char* mcpu_status_string(mcpu_status s) {
  switch (s) {
    case MCPU_OK: return "ok";
    case MCPU_ERR_INVALID_ARG: return "invalid argument";
    case MCPU_ERR_UNSUPPORTED: return "unsupported configuration";
    case MCPU_ERR_WORKSPACE_TOO_SMALL: return "workspace too small";
    case MCPU_ERR_CUDA: return "CUDA runtime error";
    case MCPU_ERR_BAD_PAGE: return "block table names a page outside the pool";
    case MCPU_ERR_BAD_LENGTHS: return "inconsistent seq_lens / query_start_loc";
    case MCPU_ERR_TIMEOUT: return "device wait timed out";
    case MCPU_ERR_INTERNAL: return "work plan exceeded its bound";
    case MCPU_ERR_POOL_EXHAUSTED: return "no free KV page left";
    case MCPU_ERR_UNSUPPORTED_ROW: return "a row this variant does not handle was skipped";
  }
  return "unknown status";
}

size_t mcpu_workspace_size(const mcpu_dims* dims) {
  if (check_dims(dims) != MCPU_OK) return 0;
  const int g = dims->num_q_heads / dims->num_kv_heads;
  return workspace_layout(dims->num_seqs, dims->total_q, dims->num_q_heads, g).total;
}

mcpu_status mcpu_kv_append(const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                           const int32_t* block_table, const int32_t* seq_lens, const int32_t* query_start_loc,
                           const mcpu_dims* dims, int32_t* status_word, mcpu_stream_t stream) {
  mcpu_status st = check_dims(dims);
  if (st != MCPU_OK) return st;
  if (dims->total_q == 0 || dims->num_seqs == 0) return MCPU_OK;
  if (!k_new || !v_new || !k_cache || !v_cache || !block_table || !seq_lens || !query_start_loc || !status_word)
    return MCPU_ERR_INVALID_ARG;
  if (!aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) ||
      !aligned(block_table, 4) || !aligned(seq_lens, 4) || !aligned(query_start_loc, 4) || !aligned(status_word, 4))
    return MCPU_ERR_INVALID_ARG;
  if (dims->num_pages < 1 || dims->max_pages_per_seq < 1) return MCPU_ERR_INVALID_ARG;
  DeviceState* dev = nullptr;  // one-time per-device kernel setup
  st = device_state(&dev);
  if (st != MCPU_OK) return st;
  return from_cuda(launch_kv_append(k_new, v_new, k_cache, v_cache, block_table, seq_lens, query_start_loc,
                                    status_word, dims->num_seqs, dims->total_q, dims->max_pages_per_seq,
                                    dims->num_pages, dims->num_kv_heads, reinterpret_cast<cudaStream_t>(stream)));
}

mcpu_status mcpu_rope_kv_append(void* q, const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                                const int32_t* block_table, const int32_t* seq_lens,
                                const int32_t* query_start_loc, const float* cos_sin, int32_t max_position,
                                const mcpu_dims* dims, int32_t* status_word, mcpu_stream_t stream) {
  mcpu_status st = check_dims(dims);
  if (st != MCPU_OK) return st;
  if (dims->total_q == 0 || dims->num_seqs == 0) return MCPU_OK;
  if (!q || !k_new || !v_new || !k_cache || !v_cache || !block_table || !seq_lens || !query_start_loc ||
      !cos_sin || !status_word || max_position < 1)
    return MCPU_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(k_cache, 16) ||
      !aligned(v_cache, 16) || !aligned(cos_sin, 4) || !aligned(status_word, 4))
    return MCPU_ERR_INVALID_ARG;
  if (dims->num_pages < 1 || dims->max_pages_per_seq < 1) return MCPU_ERR_INVALID_ARG;
  DeviceState* dev = nullptr;
  st = device_state(&dev);
  if (st != MCPU_OK) return st;
  return from_cuda(launch_rope_append(q, k_new, v_new, k_cache, v_cache, block_table, seq_lens, query_start_loc,
                                      cos_sin, max_position, status_word, dims->num_seqs, dims->total_q,
                                      dims->max_pages_per_seq, dims->num_pages, dims->num_q_heads,
                                      dims->num_kv_heads, reinterpret_cast<cudaStream_t>(stream)));
}

mcpu_status mcpu_grow_block_tables(int32_t* block_table, const int32_t* seq_lens, const mcpu_dims* dims,
                                   const int32_t* free_pages, int32_t* free_count, int32_t* status_word,
                                   mcpu_stream_t stream) {
  if (!dims || dims->num_seqs < 0 || dims->max_pages_per_seq < 0) return MCPU_ERR_INVALID_ARG;
  if (dims->num_seqs == 0) return MCPU_OK;
  if (!block_table || !seq_lens || !free_pages || !free_count || !status_word) return MCPU_ERR_INVALID_ARG;
  if (!aligned(block_table, 4) || !aligned(seq_lens, 4) || !aligned(free_pages, 4) || !aligned(free_count, 4) ||
      !aligned(status_word, 4))
    return MCPU_ERR_INVALID_ARG;
  return from_cuda(launch_grow_tables(block_table, seq_lens, dims->num_seqs, dims->max_pages_per_seq, free_pages,
                                      free_count, status_word, reinterpret_cast<cudaStream_t>(stream)));
}

mcpu_status mcpu_paged_attention_forward(const void* q, const void* k_cache, const void* v_cache,
                                         const int32_t* block_table, const int32_t* seq_lens,
                                         const int32_t* query_start_loc, int32_t sliding_window, float softmax_scale,
                                         const mcpu_dims* dims, void* out, float* lse, void* workspace,
                                         size_t workspace_bytes, const mcpu_options* opts, mcpu_stream_t stream) {
  mcpu_status st = check_dims(dims);
  if (st != MCPU_OK) return st;
  if (!(softmax_scale > 0.f) || softmax_scale > 3.0e38f) return MCPU_ERR_INVALID_ARG;
  if (!workspace) return MCPU_ERR_INVALID_ARG;
  if (workspace_bytes < mcpu_workspace_size(dims)) return MCPU_ERR_WORKSPACE_TOO_SMALL;
  if (!aligned(workspace, 256)) return MCPU_ERR_INVALID_ARG;
  if (dims->total_q == 0 || dims->num_seqs == 0) return MCPU_OK;
  if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !query_start_loc || !out || !lse)
    return MCPU_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) || !aligned(lse, 4) ||
      !aligned(block_table, 4) || !aligned(seq_lens, 4) || !aligned(query_start_loc, 4))
    return MCPU_ERR_INVALID_ARG;
  if (dims->num_pages < 1 || dims->max_pages_per_seq < 1) return MCPU_ERR_INVALID_ARG;
  if (opts && opts->split_pages < 0) return MCPU_ERR_INVALID_ARG;
  if (opts && opts->sinks && !aligned(opts->sinks, 4)) return MCPU_ERR_INVALID_ARG;

  DeviceState* dev = nullptr;
  st = device_state(&dev);
  if (st != MCPU_OK) return st;

  const int64_t rows = (int64_t)dims->num_pages * dims->num_kv_heads * kPage;
  const bool legacy_append = opts && (opts->flags & MCPU_FLAG_MMA_SYNC_APPEND);
  const int group = dims->num_q_heads / dims->num_kv_heads;
  CUtensorMap kmap, vmap, qmap;
  if (!encode_pool(&kmap, k_cache, rows) || !encode_pool(&vmap, v_cache, rows)) return MCPU_ERR_INVALID_ARG;
  if (!legacy_append && !encode_query(&qmap, q, dims->total_q, dims->num_q_heads, group)) return MCPU_ERR_INVALID_ARG;

  AttnParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.block_table = block_table;
  p.seq_lens = seq_lens;
  p.qsl = query_start_loc;
  p.out = static_cast<__nv_bfloat16*>(out);
  p.lse = lse;
  p.ws = static_cast<uint8_t*>(workspace);
  p.num_seqs = dims->num_seqs;
  p.total_q = dims->total_q;
  p.max_pages = dims->max_pages_per_seq;
  p.num_pages = dims->num_pages;
  p.num_q_heads = dims->num_q_heads;
  p.num_kv_heads = dims->num_kv_heads;
  p.group = dims->num_q_heads / dims->num_kv_heads;
  p.lay = workspace_layout(p.num_seqs, p.total_q, p.num_q_heads, p.group);
  p.window = sliding_window > 0 ? sliding_window : 0;
  p.scale_log2 = softmax_scale * 1.4426950408889634f;
  p.total_warps_hint = dev->sms * dev->bpsm_decode * 4;
  p.forced_split_pages = opts ? opts->split_pages : 0;
  p.cascade_enabled = (opts && (opts->flags & MCPU_FLAG_NO_CASCADE)) ? 0 : 1;
  p.oob_row = (int32_t)rows;
  p.append_tile_tok = (legacy_append ? kAppendRowsMin : kAppendTcRows) / p.group;
  p.sinks = opts ? opts->sinks : nullptr;
  p.decode_only = 0;

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  void* const* ev = opts ? opts->phase_events : nullptr;
  // Under stream capture the phase events become event-record nodes of the
  // graph (recorded at every replay); otherwise plain event records.
  cudaStreamCaptureStatus capturing = cudaStreamCaptureStatusNone;
  if (ev) {
    const cudaError_t ce = cudaStreamIsCapturing(reinterpret_cast<cudaStream_t>(stream), &capturing);
    if (ce != cudaSuccess) return cuda_fail(ce);
  }
  const unsigned int rec_flags = capturing == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : 0u;
  auto mark = [&](int i, cudaStream_t on) -> cudaError_t {
    return ev ? cudaEventRecordWithFlags(reinterpret_cast<cudaEvent_t>(ev[i]), on, rec_flags) : cudaSuccess;
  };
  const bool serial = opts && (opts->flags & MCPU_FLAG_SERIAL);
  // out and lse in page-locked host memory: the append kernel's form that
  // writes whole rows over the host link
  const bool out_host = opts && (opts->flags & MCPU_FLAG_HOST_OUT_DIRECT);
  const bool cascade = p.cascade_enabled && p.window == 0;
  // Programmatic launches (the planner after the prefix scan, the cascade
  // pass after the decode kernel, the merge after the cascade pass) overlap
  // a launch with the grid before it; not when phase events are recorded
  // between the kernels.
  const bool pdl = ev == nullptr;
  auto merge_grid = [&]() {
    const int want = (p.num_seqs * p.num_q_heads + 7) / 8;
    return want < dev->sms * 8 ? (want > 0 ? want : 1) : dev->sms * 8;
  };
  auto launch_append_kernel = [&]() -> cudaError_t {
    if (legacy_append) return launch_append(kmap, vmap, p, dev->sms * dev->bpsm_append, s);
    return launch_append_tc(kmap, vmap, qmap, p, dev->sms * dev->bpsm_append_tc, out_host, s);
  };
  cudaError_t e = mark(0, s);
  if (e == cudaSuccess) e = launch_plan(p, s, pdl);
  if (e == cudaSuccess) e = mark(1, s);
  if (serial) {
    if (e == cudaSuccess) e = launch_decode(kmap, vmap, p, dev->sms * dev->bpsm_decode, false, s, false);
    if (e == cudaSuccess) e = mark(2, s);
    if (e == cudaSuccess && cascade) e = launch_decode(kmap, vmap, p, dev->sms * dev->bpsm_cascade, true, s, pdl);
    if (e == cudaSuccess) e = mark(3, s);
    if (e == cudaSuccess) e = launch_append_kernel();
    if (e == cudaSuccess) e = mark(4, s);
    if (e == cudaSuccess) e = launch_merge(p, merge_grid(), s, false);
  } else {
    // fork: the append kernel goes first on `stream` (its CTAs claim the
    // SMs); the decode kernel follows on the low-priority side stream and its
    // CTAs (few registers) fill the room each SM has left. The cascade pass
    // comes after decode on the side stream: its CTAs need more registers
    // than an SM running an append CTA has free, so it may only start as the
    // append kernel drains. The merge, which reads only decode and cascade
    // partials and writes only split decode rows, ends the side stream's
    // chain, so it can run while the append kernel still does. Join last.
    std::lock_guard<std::mutex> lock(dev->fork_mu);
    if (e == cudaSuccess) e = cudaEventRecord(dev->ev_fork, s);
    if (e == cudaSuccess) e = launch_append_kernel();
    if (e == cudaSuccess) e = mark(4, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(dev->side, dev->ev_fork, 0);
    if (e == cudaSuccess) e = launch_decode(kmap, vmap, p, dev->sms * dev->bpsm_decode, false, dev->side, false);
    if (e == cudaSuccess) e = mark(2, dev->side);
    if (e == cudaSuccess && cascade)
      e = launch_decode(kmap, vmap, p, dev->sms * dev->bpsm_cascade, true, dev->side, pdl);
    if (e == cudaSuccess) e = mark(3, dev->side);
    if (e == cudaSuccess) e = launch_merge(p, merge_grid(), dev->side, pdl);
    if (e == cudaSuccess) e = cudaEventRecord(dev->ev_join, dev->side);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, dev->ev_join, 0);
  }
  if (e == cudaSuccess) e = mark(5, s);
  return from_cuda(e);
}

mcpu_status mcpu_kv_append_fp8(const void* k_new, const void* v_new, void* kv8, const int32_t* block_table,
                               const int32_t* seq_lens, const int32_t* query_start_loc, const mcpu_dims* dims,
                               int32_t* status_word, mcpu_stream_t stream) {
  mcpu_status st = check_dims(dims);
  if (st != MCPU_OK) return st;
  if (dims->total_q == 0 || dims->num_seqs == 0) return MCPU_OK;
  if (!k_new || !v_new || !kv8 || !block_table || !seq_lens || !query_start_loc || !status_word)
    return MCPU_ERR_INVALID_ARG;
  if (!aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(kv8, 16) || !aligned(block_table, 4) ||
      !aligned(seq_lens, 4) || !aligned(query_start_loc, 4) || !aligned(status_word, 4))
    return MCPU_ERR_INVALID_ARG;
  if (dims->num_pages < 1 || dims->max_pages_per_seq < 1) return MCPU_ERR_INVALID_ARG;
  DeviceState* dev = nullptr;
  st = device_state(&dev);
  if (st != MCPU_OK) return st;
  return from_cuda(launch_kv_append_fp8(k_new, v_new, kv8, block_table, seq_lens, query_start_loc, status_word,
                                        dims->num_seqs, dims->total_q, dims->max_pages_per_seq, dims->num_pages,
                                        dims->num_kv_heads, reinterpret_cast<cudaStream_t>(stream)));
}

mcpu_status mcpu_paged_attention_forward_fp8(const void* q, const void* kv8, const int32_t* block_table,
                                             const int32_t* seq_lens, const int32_t* query_start_loc,
                                             int32_t sliding_window, float softmax_scale, const mcpu_dims* dims,
                                             void* out, float* lse, void* workspace, size_t workspace_bytes,
                                             const mcpu_options* opts, mcpu_stream_t stream) {
  mcpu_status st = check_dims(dims);
  if (st != MCPU_OK) return st;
  if (!(softmax_scale > 0.f) || softmax_scale > 3.0e38f) return MCPU_ERR_INVALID_ARG;
  if (!workspace) return MCPU_ERR_INVALID_ARG;
  if (workspace_bytes < mcpu_workspace_size(dims)) return MCPU_ERR_WORKSPACE_TOO_SMALL;
  if (!aligned(workspace, 256)) return MCPU_ERR_INVALID_ARG;
  if (dims->total_q == 0 || dims->num_seqs == 0) return MCPU_OK;
  // decode rows only: more query tokens than rows means some row appends
  if (dims->total_q > dims->num_seqs) return MCPU_ERR_UNSUPPORTED;
  if (!q || !kv8 || !block_table || !seq_lens || !query_start_loc || !out || !lse) return MCPU_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(kv8, 16) || !aligned(out, 16) || !aligned(lse, 4) || !aligned(block_table, 4) ||
      !aligned(seq_lens, 4) || !aligned(query_start_loc, 4))
    return MCPU_ERR_INVALID_ARG;
  if (dims->num_pages < 1 || dims->max_pages_per_seq < 1) return MCPU_ERR_INVALID_ARG;
  if (opts && opts->split_pages < 0) return MCPU_ERR_INVALID_ARG;
  if (opts && opts->sinks && !aligned(opts->sinks, 4)) return MCPU_ERR_INVALID_ARG;
  if (opts && (opts->flags & MCPU_FLAG_MMA_SYNC_APPEND)) return MCPU_ERR_UNSUPPORTED;

  DeviceState* dev = nullptr;
  st = device_state(&dev);
  if (st != MCPU_OK) return st;

  AttnParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.block_table = block_table;
  p.seq_lens = seq_lens;
  p.qsl = query_start_loc;
  p.out = static_cast<__nv_bfloat16*>(out);
  p.lse = lse;
  p.ws = static_cast<uint8_t*>(workspace);
  p.num_seqs = dims->num_seqs;
  p.total_q = dims->total_q;
  p.max_pages = dims->max_pages_per_seq;
  p.num_pages = dims->num_pages;
  p.num_q_heads = dims->num_q_heads;
  p.num_kv_heads = dims->num_kv_heads;
  p.group = dims->num_q_heads / dims->num_kv_heads;
  p.lay = workspace_layout(p.num_seqs, p.total_q, p.num_q_heads, p.group);
  p.window = sliding_window > 0 ? sliding_window : 0;
  p.scale_log2 = softmax_scale * 1.4426950408889634f;
  p.total_warps_hint = dev->sms * dev->bpsm_fp8 * 4;
  p.forced_split_pages = opts ? opts->split_pages : 0;
  p.cascade_enabled = (opts && (opts->flags & MCPU_FLAG_NO_CASCADE)) ? 0 : 1;
  p.oob_row = 0;
  p.append_tile_tok = kAppendTcRows / p.group;
  p.sinks = opts ? opts->sinks : nullptr;
  p.decode_only = 1;

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  void* const* ev = opts ? opts->phase_events : nullptr;
  cudaStreamCaptureStatus capturing = cudaStreamCaptureStatusNone;
  if (ev) {
    const cudaError_t ce = cudaStreamIsCapturing(s, &capturing);
    if (ce != cudaSuccess) return cuda_fail(ce);
  }
  const unsigned int rec_flags = capturing == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : 0u;
  auto mark = [&](int i) -> cudaError_t {
    return ev ? cudaEventRecordWithFlags(reinterpret_cast<cudaEvent_t>(ev[i]), s, rec_flags) : cudaSuccess;
  };
  const bool cascade = p.cascade_enabled && p.window == 0;
  // every kernel on `stream`: there is no append kernel to run beside; the
  // planner, the cascade pass and the merge are programmatic launches
  // unless phase events are recorded between the kernels
  const bool pdl = ev == nullptr;
  cudaError_t e = mark(0);
  if (e == cudaSuccess) e = launch_plan(p, s, pdl);
  if (e == cudaSuccess) e = mark(1);
  if (e == cudaSuccess) e = launch_decode_fp8(kv8, p, dev->sms * dev->bpsm_fp8, false, s, false);
  if (e == cudaSuccess) e = mark(2);
  if (e == cudaSuccess && cascade)
    e = launch_decode_fp8(kv8, p, dev->sms * dev->bpsm_fp8_cascade, true, s, pdl);
  if (e == cudaSuccess) e = mark(3);
  if (e == cudaSuccess) e = mark(4);
  if (e == cudaSuccess) {
    const int want = (p.num_seqs * p.num_q_heads + 7) / 8;
    const int grid = want < dev->sms * 8 ? (want > 0 ? want : 1) : dev->sms * 8;
    e = launch_merge(p, grid, s, pdl);
  }
  if (e == cudaSuccess) e = mark(5);
  return from_cuda(e);
}

mcpu_status mcpu_selftest_append_abort(const void* q, const void* k_cache, const void* v_cache,
                                       const int32_t* block_table, const int32_t* seq_lens,
                                       const int32_t* query_start_loc, float softmax_scale, const mcpu_dims* dims,
                                       void* out, float* lse, void* workspace, size_t workspace_bytes,
                                       int32_t stall_role, int64_t* report, mcpu_stream_t stream) {
  mcpu_status st = check_dims(dims);
  if (st != MCPU_OK) return st;
  if (stall_role < 0 || stall_role > 2) return MCPU_ERR_INVALID_ARG;
  if (!report || !aligned(report, 8)) return MCPU_ERR_INVALID_ARG;
  if (!(softmax_scale > 0.f) || softmax_scale > 3.0e38f) return MCPU_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256)) return MCPU_ERR_INVALID_ARG;
  if (workspace_bytes < mcpu_workspace_size(dims)) return MCPU_ERR_WORKSPACE_TOO_SMALL;
  if (dims->total_q == 0 || dims->num_seqs == 0) return MCPU_ERR_INVALID_ARG;
  if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !query_start_loc || !out || !lse)
    return MCPU_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) || !aligned(lse, 4) ||
      !aligned(block_table, 4) || !aligned(seq_lens, 4) || !aligned(query_start_loc, 4))
    return MCPU_ERR_INVALID_ARG;
  if (dims->num_pages < 1 || dims->max_pages_per_seq < 1) return MCPU_ERR_INVALID_ARG;
  DeviceState* dev = nullptr;
  st = device_state(&dev);
  if (st != MCPU_OK) return st;
  const int64_t rows = (int64_t)dims->num_pages * dims->num_kv_heads * kPage;
  const int group = dims->num_q_heads / dims->num_kv_heads;
  CUtensorMap kmap, vmap, qmap;
  if (!encode_pool(&kmap, k_cache, rows) || !encode_pool(&vmap, v_cache, rows) ||
      !encode_query(&qmap, q, dims->total_q, dims->num_q_heads, group))
    return MCPU_ERR_INVALID_ARG;
  AttnParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.block_table = block_table;
  p.seq_lens = seq_lens;
  p.qsl = query_start_loc;
  p.out = static_cast<__nv_bfloat16*>(out);
  p.lse = lse;
  p.ws = static_cast<uint8_t*>(workspace);
  p.num_seqs = dims->num_seqs;
  p.total_q = dims->total_q;
  p.max_pages = dims->max_pages_per_seq;
  p.num_pages = dims->num_pages;
  p.num_q_heads = dims->num_q_heads;
  p.num_kv_heads = dims->num_kv_heads;
  p.group = group;
  p.lay = workspace_layout(p.num_seqs, p.total_q, p.num_q_heads, p.group);
  p.window = 0;
  p.scale_log2 = softmax_scale * 1.4426950408889634f;
  p.total_warps_hint = dev->sms * dev->bpsm_decode * 4;
  p.forced_split_pages = 0;
  p.cascade_enabled = 0;
  p.oob_row = (int32_t)rows;
  p.append_tile_tok = kAppendTcRows / p.group;
  p.sinks = nullptr;
  p.decode_only = 0;
  p.selftest_stall = stall_role;
  p.selftest_report = report;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(report, 0, 16 * sizeof(int64_t), s);
  if (e == cudaSuccess) e = launch_plan(p, s, false);
  if (e == cudaSuccess) e = launch_append_tc_selftest(kmap, vmap, qmap, p, s);
  return from_cuda(e);
}

mcpu_status mcpu_read_device_status(const void* workspace, mcpu_stream_t stream, int32_t* status_bits) {
  if (!workspace) return MCPU_ERR_INVALID_ARG;
  int32_t bits = 0;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&bits, workspace, sizeof(bits), cudaMemcpyDeviceToHost, s) != cudaSuccess) return MCPU_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return MCPU_ERR_CUDA;
  if (status_bits) *status_bits = bits;
  if (bits & kStatusTimeout) return MCPU_ERR_TIMEOUT;
  if (bits & kStatusBadPage) return MCPU_ERR_BAD_PAGE;
  if (bits & kStatusBadLengths) return MCPU_ERR_BAD_LENGTHS;
  if (bits & kStatusPlanOverflow) return MCPU_ERR_INTERNAL;
  if (bits & kStatusPoolExhausted) return MCPU_ERR_POOL_EXHAUSTED;
  if (bits & kStatusUnsupportedRow) return MCPU_ERR_UNSUPPORTED_ROW;
  return MCPU_OK;
}

mcpu_status mcpu_reset_device_status(void* workspace, mcpu_stream_t stream) {
  if (!workspace) return MCPU_ERR_INVALID_ARG;
  return from_cuda(cudaMemsetAsync(workspace, 0, sizeof(int32_t), reinterpret_cast<cudaStream_t>(stream)));
}

}  // extern "C"
