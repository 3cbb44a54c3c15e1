// Fused rotary embedding + KV append, and device-side growth of block tables.
//
// rope_append_kernel: for every query token t of row r at position
// p = S_r - L_r + i, rotates q[t] (all q heads, in place) and k_new[t] (all
// kv heads) by the angles of table row p, then writes the rotated k and the
// unrotated v into the row's page, as the plain KV append does. The rotation
// pairs dimension i with i + D/2 (half split):
//   y_i = x_i cos_i(p) - x_{i+D/2} sin_i(p),  y_{i+D/2} = x_{i+D/2} cos_i(p) + x_i sin_i(p)
// in fp32, rounded once to bf16. One warp handles one 64-dim row: lane l owns
// dims l and l + 32.
//
// grow_tables_kernel: every logical page a row needs for its S_r tokens and
// whose block-table entry is negative gets a page popped from a device stack
// of free page ids; entries already set (shared prompt pages, earlier pages)
// are left alone. An empty stack sets kStatusPoolExhausted.
#include "common.cuh"

namespace mcpu {

constexpr int kRopeWarps = 8;

struct RopeParams {
  __nv_bfloat16* q;
  const __nv_bfloat16* k_new;
  const __nv_bfloat16* v_new;
  __nv_bfloat16* k_cache;
  __nv_bfloat16* v_cache;
  const int32_t* block_table;
  const int32_t* seq_lens;
  const int32_t* qsl;
  const float* cos_sin;  // [max_position, 64]: cos then sin
  int32_t* status;
  int32_t num_seqs, total_q, max_pages, num_pages, num_q_heads, num_kv_heads, max_position;
};

// one CTA per query token: warps loop over the q heads, then k, then v rows
__global__ void __launch_bounds__(kRopeWarps * 32) rope_append_kernel(const RopeParams p) {
  const int t = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ int s_pos, s_dst;  // position (-1: skip), destination page * 16 + slot (-1: none)
  if (threadIdx.x == 0) {
    int pos = -1, dst = -1;
    if (p.qsl[0] != 0 || p.qsl[p.num_seqs] != p.total_q) {
      atomicOr(p.status, kStatusBadLengths);
    } else {
      int lo = 0, hi = p.num_seqs;  // qsl[lo] <= t < qsl[hi]
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(p.qsl + mid) <= t) lo = mid; else hi = mid;
      }
      const int q0 = __ldg(p.qsl + lo), q1 = __ldg(p.qsl + lo + 1);
      const int L = q1 - q0, S = __ldg(p.seq_lens + lo);
      if (L < 1 || S < L || S > p.max_pages * kPage || t < q0 || t >= q1) {
        atomicOr(p.status, kStatusBadLengths);
      } else {
        pos = S - L + (t - q0);
        if (pos >= p.max_position) {
          atomicOr(p.status, kStatusBadLengths);
          pos = -1;
        } else {
          const int page = __ldg(p.block_table + (size_t)lo * p.max_pages + pos / kPage);
          if (page < 0 || page >= p.num_pages)
            atomicOr(p.status, kStatusBadPage);
          else
            dst = page * kPage + pos % kPage;
        }
      }
    }
    s_pos = pos;
    s_dst = dst;
  }
  __syncthreads();
  const int pos = s_pos, dst = s_dst;
  if (pos < 0) return;
  const float c = __ldg(p.cos_sin + (size_t)pos * kHeadDim + lane);
  const float s = __ldg(p.cos_sin + (size_t)pos * kHeadDim + 32 + lane);
  const int Hq = p.num_q_heads, Hkv = p.num_kv_heads;
  for (int row = warp; row < Hq + 2 * Hkv; row += kRopeWarps) {
    if (row < Hq) {  // q, rotated in place
      __nv_bfloat16* x = p.q + ((size_t)t * Hq + row) * kHeadDim;
      const float a = __bfloat162float(x[lane]), b = __bfloat162float(x[lane + 32]);
      __syncwarp();
      x[lane] = __float2bfloat16_rn(a * c - b * s);
      x[lane + 32] = __float2bfloat16_rn(b * c + a * s);
    } else if (dst >= 0) {
      const bool is_k = row < Hq + Hkv;
      const int h = is_k ? row - Hq : row - Hq - Hkv;
      const __nv_bfloat16* x = (is_k ? p.k_new : p.v_new) + ((size_t)t * Hkv + h) * kHeadDim;
      __nv_bfloat16* out = (is_k ? p.k_cache : p.v_cache) +
                           (((size_t)(dst / kPage) * Hkv + h) * kPage + dst % kPage) * kHeadDim;
      if (is_k) {
        const float a = __bfloat162float(x[lane]), b = __bfloat162float(x[lane + 32]);
        out[lane] = __float2bfloat16_rn(a * c - b * s);
        out[lane + 32] = __float2bfloat16_rn(b * c + a * s);
      } else {
        out[lane] = x[lane];
        out[lane + 32] = x[lane + 32];
      }
    }
  }
}

cudaError_t launch_rope_append(void* q, const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                               const int32_t* block_table, const int32_t* seq_lens, const int32_t* qsl,
                               const float* cos_sin, int32_t max_position, int32_t* status, int32_t num_seqs,
                               int32_t total_q, int32_t max_pages, int32_t num_pages, int32_t num_q_heads,
                               int32_t num_kv_heads, cudaStream_t stream) {
  RopeParams p;
  p.q = static_cast<__nv_bfloat16*>(q);
  p.k_new = static_cast<const __nv_bfloat16*>(k_new);
  p.v_new = static_cast<const __nv_bfloat16*>(v_new);
  p.k_cache = static_cast<__nv_bfloat16*>(k_cache);
  p.v_cache = static_cast<__nv_bfloat16*>(v_cache);
  p.block_table = block_table;
  p.seq_lens = seq_lens;
  p.qsl = qsl;
  p.cos_sin = cos_sin;
  p.status = status;
  p.num_seqs = num_seqs;
  p.total_q = total_q;
  p.max_pages = max_pages;
  p.num_pages = num_pages;
  p.num_q_heads = num_q_heads;
  p.num_kv_heads = num_kv_heads;
  p.max_position = max_position;
  rope_append_kernel<<<total_q, kRopeWarps * 32, 0, stream>>>(p);
  return cudaGetLastError();
}

// one warp per row: lanes take the row's logical pages 32 at a time
__global__ void __launch_bounds__(256) grow_tables_kernel(int32_t* block_table, const int32_t* seq_lens,
                                                          int32_t num_seqs, int32_t max_pages,
                                                          const int32_t* free_pages, int32_t* free_count,
                                                          int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (r >= num_seqs) return;
  const int S = seq_lens[r];
  if (S < 0 || S > max_pages * kPage) {
    if (lane == 0) atomicOr(status, kStatusBadLengths);
    return;
  }
  const int need = (S + kPage - 1) / kPage;
  int32_t* row = block_table + (size_t)r * max_pages;
  for (int j = lane; j < need; j += 32) {
    if (row[j] >= 0) continue;
    const int top = atomicSub(free_count, 1);
    if (top <= 0) {
      atomicAdd(free_count, 1);  // give the slot back: the stack is empty
      atomicOr(status, kStatusPoolExhausted);
    } else {
      row[j] = free_pages[top - 1];
    }
  }
}

cudaError_t launch_grow_tables(int32_t* block_table, const int32_t* seq_lens, int32_t num_seqs, int32_t max_pages,
                               const int32_t* free_pages, int32_t* free_count, int32_t* status,
                               cudaStream_t stream) {
  const int warps_per_cta = 8;
  const int grid = (num_seqs + warps_per_cta - 1) / warps_per_cta;
  grow_tables_kernel<<<grid, warps_per_cta * 32, 0, stream>>>(block_table, seq_lens, num_seqs, max_pages,
                                                               free_pages, free_count, status);
  return cudaGetLastError();
}

}  // namespace mcpu
