// Log-sum-exp merge of split-KV / cascade partials.
//
// A decode row whose keys were processed in several parts (KV splits, and
// for GRPO-group members the shared-prefix part) has, per query head, parts
// i with a normalised output o_i and a base-2 log normaliser b_i. Exactly:
//   b = b_max + log2(sum_i 2^(b_i - b_max)),  out = sum_i 2^(b_i - b) o_i,
// and the reported lse is b * ln 2. An attention sink sigma adds a part
// 2^(sigma log2 e) with no value. One warp merges one (row, head); each
// lane owns two of the 64 dims. The parts' loads are issued together (their
// normalisers one per lane, their outputs four at a time), so a row costs a
// few memory round trips, not two per part; the sums still run in part
// order.
#include "common.cuh"

namespace mcpu {

constexpr int kMergeWarps = 8;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__global__ void __launch_bounds__(kMergeWarps * 32) merge_kernel(const AttnParams p) {
  // launched programmatically after the last kernel that writes partials:
  // nothing is read before that kernel (and, through its own wait, every
  // earlier one) has completed
  grid_dep_wait();
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
    // an attention sink joins the normaliser as one more part with no value
    const float s2 = sink_log2(p, h);
    // the parts' log normalisers, 32 at a time (lane i holds part base + i),
    // so that their loads are in flight together
    float bmax = s2;
    for (int base = 0; base < mr.n_parts; base += 32) {
      const int i = base + lane;
      const float b = i < mr.n_parts ? lse_part[(size_t)(mr.part_off + i) * Hq + h] : -INFINITY;
      bmax = fmaxf(bmax, warp_max(b));
    }
    float sum = s2 > -INFINITY ? fast_exp2(s2 - bmax) : 0.f, o0 = 0.f, o1 = 0.f;
    if (bmax != -INFINITY) {
      for (int base = 0; base < mr.n_parts; base += 32) {
        const int i = base + lane, cnt = min(32, mr.n_parts - base);
        const float wl = i < mr.n_parts ? fast_exp2(lse_part[(size_t)(mr.part_off + i) * Hq + h] - bmax) : 0.f;
        const float2* vp = reinterpret_cast<const float2*>(o_part + ((size_t)(mr.part_off + base) * Hq + h) * kHeadDim);
        const size_t vstride = (size_t)Hq * kHeadDim / 2;  // float2 elements from one part to the next
        // parts in order (the same sums as one part at a time), four loads in flight
        int j = 0;
        for (; j + 4 <= cnt; j += 4) {
          float2 v[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) v[u] = vp[(j + u) * vstride + lane];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float wgt = __shfl_sync(0xffffffffu, wl, j + u);
            sum += wgt;
            o0 += wgt * v[u].x;
            o1 += wgt * v[u].y;
          }
        }
        for (; j < cnt; ++j) {
          const float2 v = vp[j * vstride + lane];
          const float wgt = __shfl_sync(0xffffffffu, wl, j);
          sum += wgt;
          o0 += wgt * v.x;
          o1 += wgt * v.y;
        }
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

cudaError_t launch_merge(const AttnParams& p, int grid, cudaStream_t stream, bool programmatic) {
  LaunchCfg lc(dim3(grid), dim3(kMergeWarps * 32), 0, stream, programmatic);
  return cudaLaunchKernelEx(&lc.cfg, merge_kernel, p);
}

}  // namespace mcpu
