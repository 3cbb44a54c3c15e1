// KV append writer: every query token's new K and V rows go to
// (block_table[r][pos / 16], pos % 16) with pos = S_r - L_r + i, bit for bit.
//
// A CTA covers 64 consecutive query tokens. Warp 0 first finds each token's
// row by binary search over query_start_loc and checks the row's lengths and
// the destination page; then every (token, kv head, K|V) row of 128 bytes is
// moved by 8 threads with one 16-byte load and one 16-byte store each.
#include "common.cuh"

namespace mcpu {

constexpr int kAppendTokensPerCta = 64;
constexpr int kKvAppendThreads = 256;

struct KvAppendParams {
  const uint4* k_new;   // [T, Hkv, D] as 16-byte vectors
  const uint4* v_new;
  uint4* k_cache;       // [P, Hkv, 16, D]
  uint4* v_cache;
  const int32_t* block_table;
  const int32_t* seq_lens;
  const int32_t* qsl;
  int32_t* status;
  int32_t num_seqs, total_q, max_pages, num_pages, num_kv_heads;
};

__global__ void __launch_bounds__(kKvAppendThreads) kv_append_kernel(const KvAppendParams p) {
  __shared__ int s_dst[kAppendTokensPerCta];  // destination (page * 16 + slot), -1 = skip
  const int t0 = blockIdx.x * kAppendTokensPerCta;
  if (threadIdx.x < kAppendTokensPerCta) {
    const int t = t0 + threadIdx.x;
    int dst = -1;
    if (t < p.total_q) {
      // row r with qsl[r] <= t < qsl[r + 1]
      int lo = 0, hi = p.num_seqs;  // invariant: qsl[lo] <= t < qsl[hi]
      if (p.qsl[0] != 0 || p.qsl[p.num_seqs] != p.total_q) {
        atomicOr(p.status, kStatusBadLengths);
        hi = -1;
      }
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (__ldg(p.qsl + mid) <= t) lo = mid; else hi = mid;
      }
      if (hi > 0) {
        const int r = lo;
        const int q0 = __ldg(p.qsl + r), q1 = __ldg(p.qsl + r + 1);
        const int L = q1 - q0, S = __ldg(p.seq_lens + r);
        if (L < 1 || S < L || S > p.max_pages * kPage || t < q0 || t >= q1) {
          atomicOr(p.status, kStatusBadLengths);
        } else {
          const int pos = S - L + (t - q0);
          const int page = __ldg(p.block_table + (size_t)r * p.max_pages + pos / kPage);
          if (page < 0 || page >= p.num_pages)
            atomicOr(p.status, kStatusBadPage);
          else
            dst = page * kPage + pos % kPage;
        }
      }
    }
    s_dst[threadIdx.x] = dst;
  }
  __syncthreads();
  // 16-byte vectors per (token, kv head) row: 8; K and V: 16 per (token, head)
  const int per_tok = p.num_kv_heads * 16;
  const int n_tok = min(kAppendTokensPerCta, p.total_q - t0);
  for (int i = threadIdx.x; i < n_tok * per_tok; i += kKvAppendThreads) {
    const int tl = i / per_tok, rem = i % per_tok;
    const int h = rem >> 4, which = (rem >> 3) & 1, vec = rem & 7;
    const int dst = s_dst[tl];
    if (dst < 0) continue;
    const int page = dst / kPage, slot = dst % kPage;
    const size_t src = ((size_t)(t0 + tl) * p.num_kv_heads + h) * 8 + vec;
    const size_t dpos = (((size_t)page * p.num_kv_heads + h) * kPage + slot) * 8 + vec;
    if (which == 0)
      p.k_cache[dpos] = __ldg(p.k_new + src);
    else
      p.v_cache[dpos] = __ldg(p.v_new + src);
  }
}

cudaError_t prepare_kv_append_kernel() {
  return cudaFuncSetAttribute(kv_append_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                              cudaSharedmemCarveoutMaxShared);
}

cudaError_t launch_kv_append(const void* k_new, const void* v_new, void* k_cache, void* v_cache,
                             const int32_t* block_table, const int32_t* seq_lens, const int32_t* qsl,
                             int32_t* status, int32_t num_seqs, int32_t total_q, int32_t max_pages,
                             int32_t num_pages, int32_t num_kv_heads, cudaStream_t stream) {
  KvAppendParams p;
  p.k_new = static_cast<const uint4*>(k_new);
  p.v_new = static_cast<const uint4*>(v_new);
  p.k_cache = static_cast<uint4*>(k_cache);
  p.v_cache = static_cast<uint4*>(v_cache);
  p.block_table = block_table;
  p.seq_lens = seq_lens;
  p.qsl = qsl;
  p.status = status;
  p.num_seqs = num_seqs;
  p.total_q = total_q;
  p.max_pages = max_pages;
  p.num_pages = num_pages;
  p.num_kv_heads = num_kv_heads;
  const int grid = (total_q + kAppendTokensPerCta - 1) / kAppendTokensPerCta;
  kv_append_kernel<<<grid, kKvAppendThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace mcpu
