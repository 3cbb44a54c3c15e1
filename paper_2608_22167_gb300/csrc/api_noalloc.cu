// mcpu_paged_attention_forward_noalloc: the paged-attention forward for
// callers that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc (or any allocating routine): an
// inference engine that reserves all of a GPU's memory for its KV pool up
// front and forbids later allocations, code that runs while a stream is being
// captured into a CUDA graph, or a host process that only receives device
// pointers from another component. They cannot provide the workspace that
// mcpu_paged_attention_forward asks for. This entry point instead keeps its
// scratch (the device status word and the work plan) in a fixed-size array in
// the library's own device memory, which every GPU that loads the library
// holds until the process exits.
//
// To stay within that fixed size it runs the forward pass without the two
// features that need per-call partial results: decode rows are not split
// across SMs and the shared-prefix (cascade) pass is off. The results are the
// same attention (up to rounding); long decode rows are slower.
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
cudaError_t launch_append_tc(const CUtensorMap& kmap, const CUtensorMap& vmap, const CUtensorMap& qmap,
                             const AttnParams& p, int grid, bool out_host, cudaStream_t stream);
cudaError_t prepare_append_tc_kernel(int* bpsm);
}  // namespace mcpu

namespace {

using namespace mcpu;

// The fixed scratch: 4 MiB per device. The plan needs well under this for
// every batch the planner accepts (num_seqs <= 2048) with total_q up to
// kNoallocMaxTokens; larger requests are rejected.
constexpr size_t kNoallocScratchBytes = 4u << 20;
constexpr int32_t kNoallocMaxTokens = 262144;
__device__ __align__(256) uint8_t g_noalloc_scratch[kNoallocScratchBytes];

constexpr int kMaxDevices = 64;
struct NoallocDevice {
  bool ready = false;
  void* scratch = nullptr;  // device address of g_noalloc_scratch on this device
  int sms = 0, bpsm_decode = 0, bpsm_cascade = 0, bpsm_append_tc = 0;
};
std::mutex g_mu;
NoallocDevice g_dev[kMaxDevices];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

// Once per device, with that device current: the scratch array's device
// address (host code only sees a host-side stand-in for the symbol), the
// kernels' shared-memory limits and occupancy.
mcpu_status noalloc_device(NoallocDevice** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= kMaxDevices) return MCPU_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  NoallocDevice& d = g_dev[dev];
  if (!d.ready) {
    if (!g_encode) {
      void* fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if ((e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q)) !=
          cudaSuccess)
        return cuda_fail(e);
      if (q != cudaDriverEntryPointSuccess || fn == nullptr) return MCPU_ERR_CUDA;
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    void* ptr = nullptr;
    if ((e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch)) != cudaSuccess) return cuda_fail(e);
    if (ptr == nullptr) return MCPU_ERR_CUDA;
    if ((e = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_plan_kernel()) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_decode_kernels(&d.bpsm_decode, &d.bpsm_cascade)) != cudaSuccess) return cuda_fail(e);
    if ((e = prepare_append_tc_kernel(&d.bpsm_append_tc)) != cudaSuccess) return cuda_fail(e);
    if (d.bpsm_decode < 1 || d.bpsm_append_tc < 1) return MCPU_ERR_CUDA;
    d.scratch = ptr;
    d.ready = true;
  }
  *out = &d;
  return MCPU_OK;
}

bool encode_tiled(CUtensorMap* map, const void* base, cuuint32_t rank, const cuuint64_t* dims,
                  const cuuint64_t* strides, const cuuint32_t* box) {
  const cuuint32_t estr[3] = {1, 1, 1};
  return g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

extern "C" mcpu_status mcpu_paged_attention_forward_noalloc(
    const void* q, const void* k_cache, const void* v_cache, const int32_t* block_table, const int32_t* seq_lens,
    const int32_t* query_start_loc, int32_t sliding_window, float softmax_scale, const mcpu_dims* dims, void* out,
    float* lse, int32_t* status_word, mcpu_stream_t stream) {
  // ---- the same argument checks as mcpu_paged_attention_forward
  const mcpu_status dst = check_dims(dims);
  if (dst != MCPU_OK) return dst;
  const mcpu_dims& d = *dims;
  const int group = d.num_q_heads / d.num_kv_heads;
  if (!(softmax_scale > 0.f) || softmax_scale > 3.0e38f) return MCPU_ERR_INVALID_ARG;
  // ---- the fixed scratch must hold the plan of this batch
  if (d.total_q > kNoallocMaxTokens) return MCPU_ERR_WORKSPACE_TOO_SMALL;
  WorkspaceLayout lay = workspace_layout(d.num_seqs, d.total_q, d.num_q_heads, group);
  // no partial results: decode rows are not split and the cascade pass is off
  lay.max_parts = 0;
  lay.o_part = lay.lse_part = lay.total = lay.o_part;
  if (lay.total > kNoallocScratchBytes) return MCPU_ERR_WORKSPACE_TOO_SMALL;
  if (d.total_q == 0 || d.num_seqs == 0) return MCPU_OK;
  if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !query_start_loc || !out || !lse)
    return MCPU_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) || !aligned(lse, 4) ||
      !aligned(block_table, 4) || !aligned(seq_lens, 4) || !aligned(query_start_loc, 4) ||
      (status_word && !aligned(status_word, 4)))
    return MCPU_ERR_INVALID_ARG;
  if (d.num_pages < 1 || d.max_pages_per_seq < 1) return MCPU_ERR_INVALID_ARG;

  NoallocDevice* dev = nullptr;
  mcpu_status st = noalloc_device(&dev);
  if (st != MCPU_OK) return st;

  const int64_t rows = (int64_t)d.num_pages * d.num_kv_heads * kPage;
  CUtensorMap kmap, vmap, qmap;
  {
    const cuuint64_t pdims[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)rows};
    const cuuint64_t pstr[1] = {(cuuint64_t)kRowBytes};
    const cuuint32_t pbox[2] = {(cuuint32_t)kHeadDim, (cuuint32_t)kPage};
    const cuuint64_t qdims[3] = {(cuuint64_t)kHeadDim, (cuuint64_t)d.num_q_heads, (cuuint64_t)d.total_q};
    const cuuint64_t qstr[2] = {(cuuint64_t)kRowBytes, (cuuint64_t)kRowBytes * d.num_q_heads};
    const cuuint32_t qbox[3] = {(cuuint32_t)kHeadDim, (cuuint32_t)group, (cuuint32_t)(kAppendTcRows / group)};
    if (!encode_tiled(&kmap, k_cache, 2, pdims, pstr, pbox) || !encode_tiled(&vmap, v_cache, 2, pdims, pstr, pbox) ||
        !encode_tiled(&qmap, q, 3, qdims, qstr, qbox))
      return MCPU_ERR_INVALID_ARG;
  }

  AttnParams p;
  p.q = static_cast<const __nv_bfloat16*>(q);
  p.block_table = block_table;
  p.seq_lens = seq_lens;
  p.qsl = query_start_loc;
  p.out = static_cast<__nv_bfloat16*>(out);
  p.lse = lse;
  p.ws = static_cast<uint8_t*>(dev->scratch);
  p.lay = lay;
  p.num_seqs = d.num_seqs;
  p.total_q = d.total_q;
  p.max_pages = d.max_pages_per_seq;
  p.num_pages = d.num_pages;
  p.num_q_heads = d.num_q_heads;
  p.num_kv_heads = d.num_kv_heads;
  p.group = group;
  p.window = sliding_window > 0 ? sliding_window : 0;
  p.scale_log2 = softmax_scale * 1.4426950408889634f;
  p.total_warps_hint = dev->sms * dev->bpsm_decode * 4;
  p.forced_split_pages = 0x3fffffff;  // one split per decode row: every row writes out/lse itself
  p.cascade_enabled = 0;
  p.oob_row = (int32_t)rows;
  p.append_tile_tok = kAppendTcRows / group;
  p.sinks = nullptr;
  p.decode_only = 0;

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // The scratch keeps the previous call's contents: the status word must
  // start at zero (the planner rewrites every other field it reads).
  // Every row writes its own output, so the log-sum-exp merge is not needed.
  cudaError_t e = cudaMemsetAsync(dev->scratch, 0, sizeof(int32_t), s);
  if (e == cudaSuccess) e = launch_plan(p, s, false);
  if (e == cudaSuccess) e = launch_decode(kmap, vmap, p, dev->sms * dev->bpsm_decode, false, s, false);
  if (e == cudaSuccess) e = launch_append_tc(kmap, vmap, qmap, p, dev->sms * dev->bpsm_append_tc, false, s);
  if (e == cudaSuccess && status_word)
    e = cudaMemcpyAsync(status_word, dev->scratch, sizeof(int32_t), cudaMemcpyDeviceToDevice, s);
  return from_cuda(e);
}
