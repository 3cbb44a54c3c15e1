// Log-sum-exp merge of split-KV / cascade partials.
//
// A decode row whose keys were processed in several parts (KV splits, and
// for GRPO-group members the shared-prefix part) has, per query head, parts
// i with a normalised output o_i and a base-2 log normaliser b_i. Exactly:
//   b = b_max + log2(sum_i 2^(b_i - b_max)),  out = sum_i 2^(b_i - b) o_i,
// and the reported lse is b * ln 2. An attention sink sigma adds a part
// 2^(sigma log2 e) with no value. One warp merges one (row, head); each
// lane owns two of the 64 dims.
#include "common.cuh"

namespace mcpu {

constexpr int kMergeWarps = 8;

__global__ void __launch_bounds__(kMergeWarps * 32) merge_kernel(const AttnParams p) {
  const PlanHeader* hdr = header(p);
  const int lane = threadIdx.x & 31;
  const int Hq = p.num_q_heads;
  const int n = hdr->n_merge * Hq;
  const MergeRow* rows = reinterpret_cast<const MergeRow*>(p.ws + p.lay.merge_rows);
  const float* o_part = reinterpret_cast<const float*>(p.ws + p.lay.o_part);
  const float* lse_part = reinterpret_cast<const float*>(p.ws + p.lay.lse_part);
  for (int w = blockIdx.x * kMergeWarps + (threadIdx.x >> 5); w < n; w += gridDim.x * kMergeWarps) {
    const MergeRow mr = rows[w / Hq];
    const int h = w % Hq;
    float bmax = -INFINITY;
    for (int i = 0; i < mr.n_parts; ++i) bmax = fmaxf(bmax, lse_part[(size_t)(mr.part_off + i) * Hq + h]);
    // an attention sink joins the normaliser as one more part with no value
    const float s2 = sink_log2(p, h);
    bmax = fmaxf(bmax, s2);
    float sum = s2 > -INFINITY ? fast_exp2(s2 - bmax) : 0.f, o0 = 0.f, o1 = 0.f;
    if (bmax != -INFINITY) {
      for (int i = 0; i < mr.n_parts; ++i) {
        const size_t idx = (size_t)(mr.part_off + i) * Hq + h;
        const float wgt = fast_exp2(lse_part[idx] - bmax);
        const float2 v = reinterpret_cast<const float2*>(o_part + idx * kHeadDim)[lane];
        sum += wgt;
        o0 += wgt * v.x;
        o1 += wgt * v.y;
      }
    }
    const float inv = sum > 0.f ? 1.f / sum : 0.f;
    const size_t orow = (size_t)mr.token * Hq + h;
    reinterpret_cast<uint32_t*>(p.out + orow * kHeadDim)[lane] = pack_bf16x2(o0 * inv, o1 * inv);
    if (lane == 0) p.lse[orow] = sum > 0.f ? (bmax + __log2f(sum)) * 0.69314718055994531f : -INFINITY;
  }
}

cudaError_t prepare_merge_kernel() {
  return cudaFuncSetAttribute(merge_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                              cudaSharedmemCarveoutMaxShared);
}

cudaError_t launch_merge(const AttnParams& p, int grid, cudaStream_t stream) {
  merge_kernel<<<grid, kMergeWarps * 32, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace mcpu
