// Calls with host buffers (declared in include/mcpu.h): mcpu_kv_append and
// mcpu_paged_attention_forward on one layer whose per-token inputs and
// outputs live in host memory. The rows are cut into slices; slice s's
// inputs are copied in on the stage's input stream while slice s - 1
// computes on the caller's stream, and its outputs go out on the output
// stream while slice s + 1 computes. Two staging slots alternate between
// calls, so the next call's inputs can arrive while this one computes.
// The copy engines of a GB300 move about 210 GB/s host to device and
// 190 GB/s back, both at once, so a layer whose copies take less than its
// compute hides them except for the first slice in and the last slice out.
// With MCPU_FLAG_HOST_OUT_DIRECT and page-locked outputs the kernels write
// out and lse over the host link themselves (SM stores reach the same
// ~190 GB/s as the copy engine), so nothing is left to move after the
// call's last kernel.
#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/mcpu.h"

namespace {

constexpr int64_t kRowBytes = 64 * 2;  // one head's 64 bf16 values
// automatic slice count: two slices from this many bytes moved per call (a
// third slice costs more in the split compute than it hides on the mixed
// and rollout batches), else one
constexpr int64_t kTwoSliceBytes = 64ll << 20;

size_t round_up(size_t x) { return (x + 255) & ~(size_t)255; }

struct Slot {
  uint8_t* base = nullptr;
  uint8_t *q = nullptr, *kn = nullptr, *vn = nullptr, *out = nullptr;
  float* lse = nullptr;
  int32_t *sl = nullptr, *qsl = nullptr;  // seq_lens [max_rows]; rebased query_start_loc of every slice
  int32_t* qsl_host = nullptr;            // page-locked source of `qsl`
  cudaEvent_t free = nullptr;             // after the slot's last output copy
  cudaEvent_t meta_copied = nullptr;      // after the copy out of qsl_host
  bool used = false;
};

}  // namespace

struct mcpu_host_stage {
  int device = 0;
  int32_t max_tokens = 0, max_rows = 0, num_q_heads = 0, num_kv_heads = 0;
  Slot slot[MCPU_MAX_HOST_SLOTS];
  int slots = 0, next = 0;
  cudaStream_t in = nullptr, out = nullptr;
  cudaEvent_t ev_in[MCPU_MAX_HOST_SLICES] = {}, ev_done[MCPU_MAX_HOST_SLICES] = {};
  cudaEvent_t ev_out = nullptr;  // after the last output copy enqueued so far
  bool any_out = false;
};

namespace {

void release(mcpu_host_stage* hs) {
  // the output stream's last event follows every call's compute and copies
  if (hs->any_out) cudaEventSynchronize(hs->ev_out);
  if (hs->in) cudaStreamSynchronize(hs->in);
  if (hs->out) cudaStreamSynchronize(hs->out);
  for (Slot& s : hs->slot) {
    if (s.free) cudaEventDestroy(s.free);
    if (s.meta_copied) cudaEventDestroy(s.meta_copied);
    if (s.qsl_host) cudaFreeHost(s.qsl_host);
    if (s.base) cudaFree(s.base);
  }
  for (int i = 0; i < MCPU_MAX_HOST_SLICES; ++i) {
    if (hs->ev_in[i]) cudaEventDestroy(hs->ev_in[i]);
    if (hs->ev_done[i]) cudaEventDestroy(hs->ev_done[i]);
  }
  if (hs->ev_out) cudaEventDestroy(hs->ev_out);
  if (hs->in) cudaStreamDestroy(hs->in);
  if (hs->out) cudaStreamDestroy(hs->out);
  delete hs;
}

bool on_stage_device(const mcpu_host_stage* hs) {
  int dev = -1;
  return cudaGetDevice(&dev) == cudaSuccess && dev == hs->device;
}

// After a failure part-way through a call: the slot is released, and the
// stage's output event placed, only after everything the call enqueued on
// the input, compute and output streams (best effort, errors ignored), so
// that no later call overwrites staging that is still in use.
mcpu_status fail_after_enqueue(mcpu_host_stage* hs, Slot& sl, cudaStream_t s, mcpu_status st) {
  cudaEventRecord(hs->ev_in[0], hs->in);
  cudaStreamWaitEvent(hs->out, hs->ev_in[0], 0);
  cudaEventRecord(hs->ev_done[0], s);
  cudaStreamWaitEvent(hs->out, hs->ev_done[0], 0);
  cudaEventRecord(sl.free, hs->out);
  cudaEventRecord(hs->ev_out, hs->out);
  hs->any_out = true;
  return st;
}

}  // namespace

extern "C" {

mcpu_status mcpu_host_stage_create(int32_t max_tokens, int32_t max_rows, int32_t num_q_heads, int32_t num_kv_heads,
                                   int32_t slots, mcpu_host_stage** stage) {
  if (!stage) return MCPU_ERR_INVALID_ARG;
  *stage = nullptr;
  if (max_tokens < 1 || max_rows < 1 || num_q_heads < 1 || num_kv_heads < 1 || num_q_heads % num_kv_heads != 0 ||
      slots < 2 || slots > MCPU_MAX_HOST_SLOTS)
    return MCPU_ERR_INVALID_ARG;
  mcpu_host_stage* hs = new mcpu_host_stage;
  hs->slots = slots;
  hs->max_tokens = max_tokens;
  hs->max_rows = max_rows;
  hs->num_q_heads = num_q_heads;
  hs->num_kv_heads = num_kv_heads;
  bool ok = cudaGetDevice(&hs->device) == cudaSuccess;
  const size_t T = (size_t)max_tokens;
  const size_t q_bytes = round_up(T * num_q_heads * kRowBytes), kv_bytes = round_up(T * num_kv_heads * kRowBytes);
  const size_t lse_bytes = round_up(T * num_q_heads * 4), sl_bytes = round_up((size_t)max_rows * 4);
  const size_t qsl_count = (size_t)max_rows + MCPU_MAX_HOST_SLICES, qsl_bytes = round_up(qsl_count * 4);
  const size_t slot_bytes = 2 * q_bytes + 2 * kv_bytes + lse_bytes + sl_bytes + qsl_bytes;
  for (int i = 0; i < slots; ++i) {
    Slot& s = hs->slot[i];
    if (!ok) break;
    ok = cudaMalloc(&s.base, slot_bytes) == cudaSuccess &&
         cudaMallocHost(&s.qsl_host, qsl_count * sizeof(int32_t)) == cudaSuccess &&
         cudaEventCreateWithFlags(&s.free, cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&s.meta_copied, cudaEventDisableTiming) == cudaSuccess;
    if (!ok) break;
    uint8_t* b = s.base;
    s.q = b;
    s.out = b + q_bytes;
    s.kn = b + 2 * q_bytes;
    s.vn = s.kn + kv_bytes;
    s.lse = reinterpret_cast<float*>(s.vn + kv_bytes);
    s.sl = reinterpret_cast<int32_t*>(s.vn + kv_bytes + lse_bytes);
    s.qsl = reinterpret_cast<int32_t*>(s.vn + kv_bytes + lse_bytes + sl_bytes);
  }
  for (int i = 0; ok && i < MCPU_MAX_HOST_SLICES; ++i)
    ok = cudaEventCreateWithFlags(&hs->ev_in[i], cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&hs->ev_done[i], cudaEventDisableTiming) == cudaSuccess;
  ok = ok && cudaEventCreateWithFlags(&hs->ev_out, cudaEventDisableTiming) == cudaSuccess &&
       cudaStreamCreateWithFlags(&hs->in, cudaStreamNonBlocking) == cudaSuccess &&
       cudaStreamCreateWithFlags(&hs->out, cudaStreamNonBlocking) == cudaSuccess;
  if (!ok) {
    release(hs);
    return MCPU_ERR_CUDA;
  }
  *stage = hs;
  return MCPU_OK;
}

mcpu_status mcpu_host_stage_destroy(mcpu_host_stage* stage) {
  if (stage) release(stage);
  return MCPU_OK;
}

mcpu_status mcpu_host_stage_wait(mcpu_host_stage* stage, mcpu_stream_t stream) {
  if (!stage) return MCPU_ERR_INVALID_ARG;
  if (!stage->any_out) return MCPU_OK;
  return cudaStreamWaitEvent(reinterpret_cast<cudaStream_t>(stream), stage->ev_out, 0) == cudaSuccess
             ? MCPU_OK
             : MCPU_ERR_CUDA;
}

mcpu_status mcpu_host_stage_sync(mcpu_host_stage* stage) {
  if (!stage) return MCPU_ERR_INVALID_ARG;
  if (!stage->any_out) return MCPU_OK;
  return cudaEventSynchronize(stage->ev_out) == cudaSuccess ? MCPU_OK : MCPU_ERR_CUDA;
}

int32_t mcpu_host_slice_rows(const int32_t* query_start_loc_host, int32_t num_seqs, int32_t slices,
                             int32_t* row_begin) {
  if (!query_start_loc_host || !row_begin || num_seqs < 0 || slices < 1 || slices > MCPU_MAX_HOST_SLICES) return 0;
  if (num_seqs == 0) {
    row_begin[0] = 0;
    return 0;
  }
  const int64_t T = query_start_loc_host[num_seqs];
  int32_t n = 0;
  row_begin[0] = 0;
  for (int32_t k = 1; k < slices; ++k) {
    // the row start nearest to k / slices of the total tokens
    const int64_t target = (T * k + slices / 2) / slices;
    int32_t lo = row_begin[n] + 1, hi = num_seqs;  // first start >= target in (previous boundary, num_seqs]
    while (lo < hi) {
      const int32_t mid = lo + (hi - lo) / 2;
      if (query_start_loc_host[mid] >= target) hi = mid;
      else lo = mid + 1;
    }
    if (lo - 1 > row_begin[n] && target - query_start_loc_host[lo - 1] < query_start_loc_host[lo] - target) --lo;
    if (lo < num_seqs && query_start_loc_host[lo] > query_start_loc_host[row_begin[n]]) row_begin[++n] = lo;
  }
  row_begin[++n] = num_seqs;
  return n;
}

}  // extern "C"

namespace {

// The device-side arguments of one slice: its rows' block-table rows,
// seq_lens and rebased query_start_loc, and its tokens' staging.
struct Slice {
  mcpu_dims dims;
  const int32_t *block_table, *seq_lens, *query_start_loc;
  const void *q, *k_new, *v_new;
  void* out;
  float* lse;
  bool out_host;  // out and lse are the caller's page-locked host buffers
};

// The caller's options for a slice's forward, with MCPU_FLAG_HOST_OUT_DIRECT
// set exactly when that forward writes into host memory.
mcpu_options slice_options(const mcpu_options* opts, const Slice& c) {
  mcpu_options o = {};
  if (opts) o = *opts;
  o.flags = c.out_host ? (o.flags | MCPU_FLAG_HOST_OUT_DIRECT) : (o.flags & ~MCPU_FLAG_HOST_OUT_DIRECT);
  return o;
}

// The pipeline shared by the bf16 and fp8 calls: checks, slicing, the
// copies in and out on the stage's streams, and `compute(slice)` (the KV
// append and forward of one slice, enqueued on `stream`) in between.
template <typename Compute>
mcpu_status host_call(mcpu_host_stage* hs, const void* q_host, const void* k_new_host, const void* v_new_host,
                      const int32_t* block_table, const int32_t* seq_lens_host,
                      const int32_t* query_start_loc_host, float softmax_scale, const mcpu_dims* dims,
                      void* out_host, float* lse_host, void* workspace, size_t workspace_bytes, int32_t slices,
                      bool out_direct_wanted, mcpu_stream_t stream, Compute compute) {
  if (!hs || !dims || !seq_lens_host || !query_start_loc_host) return MCPU_ERR_INVALID_ARG;
  if (!on_stage_device(hs)) return MCPU_ERR_INVALID_ARG;
  const int32_t B = dims->num_seqs, T = dims->total_q;
  if (B < 0 || T < 0 || B > hs->max_rows || T > hs->max_tokens || dims->num_q_heads != hs->num_q_heads ||
      dims->num_kv_heads != hs->num_kv_heads || dims->head_dim != 64)
    return MCPU_ERR_INVALID_ARG;
  if (slices < 0 || slices > MCPU_MAX_HOST_SLICES) return MCPU_ERR_INVALID_ARG;
  // the copies follow query_start_loc_host: it must run from 0 to T without decreasing
  if (query_start_loc_host[0] != 0 || query_start_loc_host[B] != T) return MCPU_ERR_INVALID_ARG;
  for (int32_t r = 0; r < B; ++r)
    if (query_start_loc_host[r + 1] < query_start_loc_host[r]) return MCPU_ERR_INVALID_ARG;
  // the wrapped calls' own checks, on the whole batch, before anything is enqueued
  if (!(softmax_scale > 0.f) || softmax_scale > 3.0e38f) return MCPU_ERR_INVALID_ARG;
  const size_t need = mcpu_workspace_size(dims);
  if (need == 0) return MCPU_ERR_UNSUPPORTED;
  if (!workspace || workspace_bytes < need) return workspace ? MCPU_ERR_WORKSPACE_TOO_SMALL : MCPU_ERR_INVALID_ARG;
  if (T == 0 || B == 0) return MCPU_OK;
  if (!q_host || !k_new_host || !v_new_host || !out_host || !lse_host || !block_table) return MCPU_ERR_INVALID_ARG;

  // outputs written by the kernels themselves: page-locked host memory the
  // device can address, and the caller asked for it
  uint8_t* out_direct = nullptr;
  uint8_t* lse_direct = nullptr;
  if (out_direct_wanted) {
    cudaPointerAttributes ao, al;
    if (cudaPointerGetAttributes(&ao, out_host) == cudaSuccess && ao.type == cudaMemoryTypeHost &&
        ao.devicePointer != nullptr && cudaPointerGetAttributes(&al, lse_host) == cudaSuccess &&
        al.type == cudaMemoryTypeHost && al.devicePointer != nullptr) {
      out_direct = static_cast<uint8_t*>(ao.devicePointer);
      lse_direct = static_cast<uint8_t*>(al.devicePointer);
    }
    (void)cudaGetLastError();  // a query of memory CUDA does not know is not an error of this call
  }

  const int64_t q_row = (int64_t)dims->num_q_heads * kRowBytes, kv_row = (int64_t)dims->num_kv_heads * kRowBytes;
  const int64_t lse_row = (int64_t)dims->num_q_heads * 4;
  // automatic slices: split only to hide copies back (the inputs of a call
  // are copied while the previous one computes)
  if (slices == 0)
    slices = (!out_direct && (int64_t)T * (2 * q_row + 2 * kv_row + lse_row) >= kTwoSliceBytes) ? 2 : 1;
  int32_t rb[MCPU_MAX_HOST_SLICES + 1];
  const int32_t n = mcpu_host_slice_rows(query_start_loc_host, B, slices, rb);

  Slot& sl = hs->slot[hs->next];
  hs->next = (hs->next + 1) % hs->slots;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // rebased query_start_loc of every slice, into the slot's page-locked
  // buffer once the copy out of it by this slot's previous call has run
  if (cudaEventSynchronize(sl.meta_copied) != cudaSuccess) return MCPU_ERR_CUDA;
  for (int32_t k = 0; k < n; ++k) {
    const int32_t a = rb[k], b = rb[k + 1], base = query_start_loc_host[a];
    for (int32_t r = a; r <= b; ++r) sl.qsl_host[a + k + (r - a)] = query_start_loc_host[r] - base;
  }
  cudaError_t e = cudaSuccess;
  if (sl.used) e = cudaStreamWaitEvent(hs->in, sl.free, 0);
  if (e == cudaSuccess) e = cudaMemcpyAsync(sl.sl, seq_lens_host, (size_t)B * 4, cudaMemcpyHostToDevice, hs->in);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(sl.qsl, sl.qsl_host, (size_t)(B + n) * 4, cudaMemcpyHostToDevice, hs->in);
  if (e == cudaSuccess) e = cudaEventRecord(sl.meta_copied, hs->in);
  sl.used = true;
  if (e != cudaSuccess) return fail_after_enqueue(hs, sl, s, MCPU_ERR_CUDA);

  const uint8_t* qh = static_cast<const uint8_t*>(q_host);
  const uint8_t* knh = static_cast<const uint8_t*>(k_new_host);
  const uint8_t* vnh = static_cast<const uint8_t*>(v_new_host);
  uint8_t* oh = static_cast<uint8_t*>(out_host);
  uint8_t* lh = reinterpret_cast<uint8_t*>(lse_host);
  for (int32_t k = 0; k < n; ++k) {
    const int32_t a = rb[k], b = rb[k + 1];
    const int64_t t0 = query_start_loc_host[a], nt = query_start_loc_host[b] - t0;
    // inputs of slice k
    e = cudaMemcpyAsync(sl.q + t0 * q_row, qh + t0 * q_row, nt * q_row, cudaMemcpyHostToDevice, hs->in);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(sl.kn + t0 * kv_row, knh + t0 * kv_row, nt * kv_row, cudaMemcpyHostToDevice, hs->in);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(sl.vn + t0 * kv_row, vnh + t0 * kv_row, nt * kv_row, cudaMemcpyHostToDevice, hs->in);
    if (e == cudaSuccess) e = cudaEventRecord(hs->ev_in[k], hs->in);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, hs->ev_in[k], 0);
    if (e != cudaSuccess) return fail_after_enqueue(hs, sl, s, MCPU_ERR_CUDA);
    // the slice's KV append and forward on the caller's stream
    Slice c;
    c.dims = *dims;
    c.dims.num_seqs = b - a;
    c.dims.total_q = (int32_t)nt;
    c.block_table = block_table + (int64_t)a * dims->max_pages_per_seq;
    c.seq_lens = sl.sl + a;
    c.query_start_loc = sl.qsl + a + k;
    c.q = sl.q + t0 * q_row;
    c.k_new = sl.kn + t0 * kv_row;
    c.v_new = sl.vn + t0 * kv_row;
    c.out = (out_direct ? out_direct : sl.out) + t0 * q_row;
    c.lse = reinterpret_cast<float*>((lse_direct ? lse_direct : reinterpret_cast<uint8_t*>(sl.lse)) + t0 * lse_row);
    c.out_host = out_direct != nullptr;
    const mcpu_status st = compute(c);
    if (st != MCPU_OK) return fail_after_enqueue(hs, sl, s, st);
    if (out_direct) continue;  // written in place by the kernels
    // its outputs, once computed
    e = cudaEventRecord(hs->ev_done[k], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(hs->out, hs->ev_done[k], 0);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(oh + t0 * q_row, sl.out + t0 * q_row, nt * q_row, cudaMemcpyDeviceToHost, hs->out);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(lh + t0 * lse_row, reinterpret_cast<uint8_t*>(sl.lse) + t0 * lse_row, nt * lse_row,
                          cudaMemcpyDeviceToHost, hs->out);
    if (e != cudaSuccess) return fail_after_enqueue(hs, sl, s, MCPU_ERR_CUDA);
  }
  if (out_direct) {  // the output stream follows the compute, as after copies
    e = cudaEventRecord(hs->ev_done[0], s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(hs->out, hs->ev_done[0], 0);
  }
  if (e == cudaSuccess) e = cudaEventRecord(sl.free, hs->out);
  if (e == cudaSuccess) e = cudaEventRecord(hs->ev_out, hs->out);
  if (e != cudaSuccess) return fail_after_enqueue(hs, sl, s, MCPU_ERR_CUDA);
  hs->any_out = true;
  return MCPU_OK;
}

}  // namespace

extern "C" {

mcpu_status mcpu_paged_attention_host(mcpu_host_stage* hs, const void* q_host, const void* k_new_host,
                                      const void* v_new_host, void* k_cache, void* v_cache,
                                      const int32_t* block_table, const int32_t* seq_lens_host,
                                      const int32_t* query_start_loc_host, int32_t sliding_window,
                                      float softmax_scale, const mcpu_dims* dims, void* out_host, float* lse_host,
                                      void* workspace, size_t workspace_bytes, const mcpu_options* opts,
                                      int32_t slices, mcpu_stream_t stream) {
  if (!k_cache || !v_cache) return MCPU_ERR_INVALID_ARG;
  int32_t* status = static_cast<int32_t*>(workspace);
  return host_call(hs, q_host, k_new_host, v_new_host, block_table, seq_lens_host, query_start_loc_host,
                   softmax_scale, dims, out_host, lse_host, workspace, workspace_bytes, slices,
                   opts && (opts->flags & MCPU_FLAG_HOST_OUT_DIRECT), stream,
                   [&](const Slice& c) {
                     mcpu_status st = mcpu_kv_append(c.k_new, c.v_new, k_cache, v_cache, c.block_table, c.seq_lens,
                                                     c.query_start_loc, &c.dims, status, stream);
                     if (st != MCPU_OK) return st;
                     const mcpu_options o = slice_options(opts, c);
                     return mcpu_paged_attention_forward(c.q, k_cache, v_cache, c.block_table, c.seq_lens,
                                                         c.query_start_loc, sliding_window, softmax_scale, &c.dims,
                                                         c.out, c.lse, workspace, workspace_bytes, &o, stream);
                   });
}

mcpu_status mcpu_paged_attention_host_fp8(mcpu_host_stage* hs, const void* q_host, const void* k_new_host,
                                          const void* v_new_host, void* kv8, const int32_t* block_table,
                                          const int32_t* seq_lens_host, const int32_t* query_start_loc_host,
                                          int32_t sliding_window, float softmax_scale, const mcpu_dims* dims,
                                          void* out_host, float* lse_host, void* workspace, size_t workspace_bytes,
                                          const mcpu_options* opts, int32_t slices, mcpu_stream_t stream) {
  if (!kv8) return MCPU_ERR_INVALID_ARG;
  int32_t* status = static_cast<int32_t*>(workspace);
  return host_call(hs, q_host, k_new_host, v_new_host, block_table, seq_lens_host, query_start_loc_host,
                   softmax_scale, dims, out_host, lse_host, workspace, workspace_bytes, slices,
                   opts && (opts->flags & MCPU_FLAG_HOST_OUT_DIRECT), stream,
                   [&](const Slice& c) {
                     mcpu_status st = mcpu_kv_append_fp8(c.k_new, c.v_new, kv8, c.block_table, c.seq_lens,
                                                         c.query_start_loc, &c.dims, status, stream);
                     if (st != MCPU_OK) return st;
                     const mcpu_options o = slice_options(opts, c);
                     return mcpu_paged_attention_forward_fp8(c.q, kv8, c.block_table, c.seq_lens, c.query_start_loc,
                                                             sliding_window, softmax_scale, &c.dims, c.out, c.lse,
                                                             workspace, workspace_bytes, &o, stream);
                   });
}

}  // extern "C"
