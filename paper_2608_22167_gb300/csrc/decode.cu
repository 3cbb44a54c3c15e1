// Split-KV paged decode and the shared-prefix (cascade) pass.
//
// One warp owns one work item: a contiguous range of pages of one kv head,
// for either one decode row (NT = 1: its g <= 8 query heads) or a cascade
// subgroup (NT = 4: up to 32 query vectors = members x g heads, all reading
// the same shared prompt pages once). Per page the warp
//   - receives the 2 KiB K block and 2 KiB V block of (page, kv head) from a
//     per-warp ring of kDecodeStages stages filled by 2-D TMA loads (128-byte
//     swizzle, so ldmatrix reads are bank-conflict free);
//   - computes S^T = K Q^T with mma.sync m16n8k16 (16 keys as M, query
//     vectors as N), masks keys outside [first_key, seq_len) on a row's
//     first and last page, and runs an online softmax in fp32 (base-2
//     exponent, scale folded in) against a lazily raised reference max;
//   - transposes P^T into the B operand with movmatrix and accumulates
//     O^T += V^T P^T (head dim as M) in fp32.
// The item ends with either the final bf16 output + lse (a decode row that
// needs one split) or a normalised fp32 partial + base-2 lse in a workspace
// slot, merged later by log-sum-exp. Warps take items from an atomic ticket.
//
// HBM traffic per (page, kv head): 4 KiB read once. Nothing else is re-read.
#include "common.cuh"

namespace mcpu {

constexpr int kDecodeWarps = 4;
constexpr int kDecodeStages = 4;
constexpr int kStageBytes = 2 * kTileBytes;  // K + V block
constexpr int kDecodeRingBytes = kDecodeStages * kStageBytes;

size_t decode_smem_bytes() {
  return 1024 /* alignment slack */ + (size_t)kDecodeWarps * kDecodeRingBytes +
         (size_t)kDecodeWarps * kDecodeStages * 8;
}

template <int NT>
__global__ void __launch_bounds__(kDecodeWarps * 32)
    decode_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                  const AttnParams p) {
  // The cascade pass (NT > 1) may be launched programmatically after the
  // decode kernel and run beside its tail: it reads nothing the decode
  // kernel writes, but it waits for that kernel before it exits, so that its
  // end still implies the decode kernel's (the merge comes after both).
  if ((NT == 1 ? header(p)->n_decode : header(p)->n_cascade) == 0) {  // nothing of this kind
    if (NT > 1) grid_dep_wait();
    return;
  }
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t ring = base + warp * kDecodeRingBytes;
  const uint32_t bars = base + kDecodeWarps * kDecodeRingBytes + warp * kDecodeStages * 8;
  float* scratch = reinterpret_cast<float*>(smem_raw + (ring - raw));

  if (lane == 0) {
    for (int s = 0; s < kDecodeStages; ++s) mbar_init(bars + 8 * s, 1);
    fence_barrier_init();
    prefetch_tensormap(&kmap);
    prefetch_tensormap(&vmap);
  }
  __syncwarp();

  const PlanHeader* hdr = header(p);
  const int Hkv = p.num_kv_heads, Hq = p.num_q_heads, g = p.group;
  const int n_items = (NT == 1 ? hdr->n_decode : hdr->n_cascade) * Hkv;
  const DecodeItem* ditems = reinterpret_cast<const DecodeItem*>(p.ws + p.lay.decode_items);
  const CascadeItem* citems = reinterpret_cast<const CascadeItem*>(p.ws + p.lay.cascade_items);
  const CascadeMember* members = reinterpret_cast<const CascadeMember*>(p.ws + p.lay.members);
  float* o_part = reinterpret_cast<float*>(p.ws + p.lay.o_part);
  float* lse_part = reinterpret_cast<float*>(p.ws + p.lay.lse_part);
  const uint64_t pol = policy_evict_first();
  const int mi = lane >> 3, ri = lane & 7;

  // Items are taken from an atomic ticket, one per warp at a time, so warps
  // that start late (their SM busy with another kernel) take fewer items.
  int* ticket = NT == 1 ? &header(p)->decode_ticket : &header(p)->cascade_ticket;
  auto next_item = [&]() -> int {
    int v = 0;
    if (lane == 0) v = atomicAdd(ticket, 1);
    return __shfl_sync(0xffffffffu, v, 0);
  };
  uint32_t seq = 0;  // pages this warp has consumed so far (ring position/phase)
  for (int it = next_item(); it < n_items; it = next_item()) {
    const int rec = it / Hkv, kvh = it % Hkv;
    int row, pb, pe, seq_len = 0, first_key = 0, slot = -1, token = 0;
    int member_off = 0, n_members = 0, split = 0;
    if (NT == 1) {
      const DecodeItem d = ditems[rec];
      row = d.row;
      pb = d.page_begin;
      pe = d.page_end;
      seq_len = d.seq_len;
      first_key = d.first_key;
      slot = d.slot;
      token = d.token;
    } else {
      const CascadeItem c = citems[rec];
      row = c.first_row;
      pb = c.page_begin;
      pe = c.page_end;
      member_off = c.member_off;
      n_members = c.n_members;
      split = c.split;
    }
    const int* bt_row = p.block_table + (size_t)row * p.max_pages;

    // Query vectors as the B operand (K = head dim, N = query vector).
    uint32_t qb[NT][4][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const int qv = nt * 8 + (lane >> 2);
      int tok = -1, head = 0;
      if (NT == 1) {
        if (qv < g) tok = token, head = kvh * g + qv;
      } else {
        const int m = qv / g;
        if (m < n_members) tok = members[member_off + m].token, head = kvh * g + qv % g;
      }
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        if (tok >= 0) {
          const uint32_t* qp = reinterpret_cast<const uint32_t*>(p.q + ((size_t)tok * Hq + head) * kHeadDim);
          qb[nt][kk][0] = __ldg(qp + kk * 8 + (lane & 3));
          qb[nt][kk][1] = __ldg(qp + kk * 8 + 4 + (lane & 3));
        } else {
          qb[nt][kk][0] = qb[nt][kk][1] = 0u;
        }
      }
    }

    // Page ids: lane i caches the id of page (chunk + i); lane 0 issues.
    const int n = pe - pb;
    int chunk_base = -32, pid_reg = 0;
    auto page_id = [&](int k) -> int {
      const int cb = k & ~31;
      if (cb != chunk_base) {
        chunk_base = cb;
        const int idx = pb + cb + lane;
        int v = -1;
        if (idx < pe) {
          v = __ldg(bt_row + idx);
          if (v < 0 || v >= p.num_pages) {
            raise_status(p, kStatusBadPage);
            v = -1;
          }
        }
        pid_reg = v;
      }
      return __shfl_sync(0xffffffffu, pid_reg, k & 31);
    };
    auto issue = [&](int k) {
      const int pid = page_id(k);
      const uint32_t s = (seq + k) % kDecodeStages;
      if (lane == 0) {
        const uint32_t bar = bars + 8 * s;
        const int y = pid < 0 ? p.oob_row : (pid * Hkv + kvh) * kPage;
        mbar_arrive_expect_tx(bar, kStageBytes);
        tma_load_2d(ring + s * kStageBytes, &kmap, 0, y, bar, pol);
        tma_load_2d(ring + s * kStageBytes + kTileBytes, &vmap, 0, y, bar, pol);
      }
    };
    const int pre = n < kDecodeStages ? n : kDecodeStages;
    for (int k = 0; k < pre; ++k) issue(k);

    // Online softmax with a lazy reference: scores are exponentiated against
    // m_ref, which is only raised (with the rescale of O and l) when a score
    // exceeds it by more than kLazy (so p <= 2^8, exact enough in bf16);
    // checking that is one warp vote per page.
    constexpr float kLazy = 8.f;
    constexpr float kNoMax = -1e30f;  // reference before the first visible key
    float m_ref[NT][2], l_run[NT][2], acc[4][NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      m_ref[nt][0] = m_ref[nt][1] = kNoMax;
      l_run[nt][0] = l_run[nt][1] = 0.f;
#pragma unroll
      for (int mt = 0; mt < 4; ++mt)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[mt][nt][e] = 0.f;
    }

    bool timed_out = false;
    for (int k = 0; k < n; ++k) {
      const uint32_t s = (seq + k) % kDecodeStages;
      const uint32_t phase = ((seq + k) / kDecodeStages) & 1u;
      const bool ok = __any_sync(0xffffffffu, mbar_wait(bars + 8 * s, phase));
      if (!ok) {
        timed_out = true;
        break;
      }
      const uint32_t kt = ring + s * kStageBytes, vt = kt + kTileBytes;

      // S^T[16 keys x 8*NT query vectors] = K Q^T
      float c[NT][4];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) c[nt][0] = c[nt][1] = c[nt][2] = c[nt][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t a0, a1, a2, a3;
        ldmatrix_x4(kt + swz128(ri + (mi & 1) * 8, 2 * kk + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(c[nt], a0, a1, a2, a3, qb[nt][kk][0], qb[nt][kk][1]);
      }

      // t = score - reference (base 2), one FFMA each
      float tv[NT][4];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) tv[nt][i] = fmaf(c[nt][i], p.scale_log2, -m_ref[nt][i & 1]);
      // keys outside [first_key, seq_len): only a row's first and last pages
      const int j0 = (pb + k) * kPage + (lane >> 2);
      const bool edge = NT == 1 && ((pb + k) * kPage < first_key || (pb + k + 1) * kPage > seq_len);
      bool v0 = true, v1 = true;
      if (edge) {
        v0 = j0 >= first_key && j0 < seq_len;
        v1 = (j0 + 8) >= first_key && (j0 + 8) < seq_len;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          tv[nt][0] = v0 ? tv[nt][0] : -INFINITY;
          tv[nt][1] = v0 ? tv[nt][1] : -INFINITY;
          tv[nt][2] = v1 ? tv[nt][2] : -INFINITY;
          tv[nt][3] = v1 ? tv[nt][3] : -INFINITY;
        }
      }
      bool over = false;
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) over |= fmaxf(fmaxf(tv[nt][0], tv[nt][2]), fmaxf(tv[nt][1], tv[nt][3])) > kLazy;
      if (__any_sync(0xffffffffu, over)) {  // rare: raise the reference to the running max
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          float sx[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) sx[i] = ((i < 2) ? v0 : v1) ? c[nt][i] * p.scale_log2 : -INFINITY;
          float mx0 = fmaxf(sx[0], sx[2]), mx1 = fmaxf(sx[1], sx[3]);
#pragma unroll
          for (int o = 4; o < 32; o <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
          }
          const float mn0 = fmaxf(m_ref[nt][0], mx0), mn1 = fmaxf(m_ref[nt][1], mx1);
          const float al0 = ex2_approx(m_ref[nt][0] - mn0), al1 = ex2_approx(m_ref[nt][1] - mn1);
          m_ref[nt][0] = mn0;
          m_ref[nt][1] = mn1;
#pragma unroll
          for (int i = 0; i < 4; ++i) tv[nt][i] = sx[i] - m_ref[nt][i & 1];
          l_run[nt][0] *= al0;
          l_run[nt][1] *= al1;
#pragma unroll
          for (int mt = 0; mt < 4; ++mt) {
            acc[mt][nt][0] *= al0;
            acc[mt][nt][1] *= al1;
            acc[mt][nt][2] *= al0;
            acc[mt][nt][3] *= al1;
          }
        }
      }
      uint32_t pb0[NT], pb1[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        const float p00 = ex2_approx(tv[nt][0]), p01 = ex2_approx(tv[nt][1]);
        const float p10 = ex2_approx(tv[nt][2]), p11 = ex2_approx(tv[nt][3]);
        l_run[nt][0] += p00 + p10;
        l_run[nt][1] += p01 + p11;
        pb0[nt] = movmatrix_trans(pack_bf16x2(p00, p01));
        pb1[nt] = movmatrix_trans(pack_bf16x2(p10, p11));
      }

      // V rows of slots outside [first_key, seq_len) were perhaps never
      // written and may hold NaN, which a zero weight does not cancel
      // (0 x NaN = NaN): on a row's first and last page they are zeroed in the
      // operand. This lane's V^T fragments a0/a1 hold keys 2c, 2c + 1 and
      // a2/a3 keys 2c + 8, 2c + 9 of the page (c = lane & 3), the lower key
      // in the low half of each word.
      uint32_t vm_lo = 0xffffffffu, vm_hi = 0xffffffffu;
      if (edge) {
        const int jv = (pb + k) * kPage + 2 * (lane & 3);
        auto seen = [&](int j) { return j >= first_key && j < seq_len; };
        vm_lo = (seen(jv) ? 0x0000ffffu : 0u) | (seen(jv + 1) ? 0xffff0000u : 0u);
        vm_hi = (seen(jv + 8) ? 0x0000ffffu : 0u) | (seen(jv + 9) ? 0xffff0000u : 0u);
      }

      // O^T[64 dims x 8*NT] += V^T P^T
#pragma unroll
      for (int mt = 0; mt < 4; ++mt) {
        uint32_t a0, a1, a2, a3;
        ldmatrix_x4_trans(vt + swz128(ri + (mi >> 1) * 8, 2 * mt + (mi & 1)), a0, a1, a2, a3);
        a0 &= vm_lo;
        a1 &= vm_lo;
        a2 &= vm_hi;
        a3 &= vm_hi;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(acc[mt][nt], a0, a1, a2, a3, pb0[nt], pb1[nt]);
      }

      // release the stage to the async proxy, then refill it
      fence_proxy_async();
      __syncwarp();
      if (k + kDecodeStages < n) issue(k + kDecodeStages);
    }
    if (timed_out) {
      raise_status(p, kStatusTimeout);
      if (NT > 1) grid_dep_wait();
      return;  // the ring's phase tracking is lost: this warp stops here
    }
    seq += n;

    // ---- epilogue: finish the row sums, stage O in shared memory
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
      for (int e = 0; e < 2; ++e)
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) l_run[nt][e] += __shfl_xor_sync(0xffffffffu, l_run[nt][e], o);
    constexpr int kLd = kHeadDim + 1;  // padded row of the staging buffer
    float* so = scratch;                        // [8*NT][kLd]
    float* sl = scratch + 8 * NT * kLd;         // [8*NT] base-2 lse
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int qv = nt * 8 + 2 * (lane & 3) + e;
        const float l = l_run[nt][e];
        const float m = l > 0.f ? m_ref[nt][e] : -INFINITY;
        float inv = l > 0.f ? 1.f / l : 0.f;
        float lse2 = l > 0.f ? m + __log2f(l) : -INFINITY;
        // a row finished here (one split) takes its sink now; split rows in the merge
        if (NT == 1 && p.sinks != nullptr && slot < 0 && qv < g)
          inv = finish_with_sink(m, l, sink_log2(p, kvh * g + qv), &lse2);
#pragma unroll
        for (int mt = 0; mt < 4; ++mt) {
          so[qv * kLd + mt * 16 + (lane >> 2)] = acc[mt][nt][e] * inv;
          so[qv * kLd + mt * 16 + (lane >> 2) + 8] = acc[mt][nt][e + 2] * inv;
        }
        if ((lane >> 2) == 0) sl[qv] = lse2;
      }
    }
    __syncwarp();
    const int n_qv = NT == 1 ? g : n_members * g;
    for (int qv = 0; qv < n_qv; ++qv) {
      const float o0 = so[qv * kLd + 2 * lane], o1 = so[qv * kLd + 2 * lane + 1];
      const float l2 = sl[qv];
      int tok, dst_slot;
      if (NT == 1) {
        tok = token;
        dst_slot = slot;
      } else {
        const CascadeMember cm = members[member_off + qv / g];
        tok = cm.token;
        dst_slot = cm.part_off + split;
      }
      const int head = kvh * g + qv % g;
      if (dst_slot < 0) {
        reinterpret_cast<uint32_t*>(p.out + ((size_t)tok * Hq + head) * kHeadDim)[lane] = pack_bf16x2(o0, o1);
        if (lane == 0) p.lse[(size_t)tok * Hq + head] = l2 * 0.69314718055994531f;
      } else {
        reinterpret_cast<float2*>(o_part + ((size_t)dst_slot * Hq + head) * kHeadDim)[lane] = make_float2(o0, o1);
        if (lane == 0) lse_part[(size_t)dst_slot * Hq + head] = l2;
      }
    }
    // the staging area is the TMA ring: order these generic accesses before
    // the next item's async-proxy writes
    fence_proxy_async();
    __syncwarp();
  }
  // no item left for this warp: the grid after this one may launch
  grid_dep_launch();
  if (NT > 1) grid_dep_wait();
}

// `programmatic` (cascade pass only): launched with programmatic stream
// serialization right after the decode kernel on the same stream.
cudaError_t launch_decode(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttnParams& p, int grid,
                          bool cascade, cudaStream_t stream, bool programmatic) {
  LaunchCfg lc(dim3(grid), dim3(kDecodeWarps * 32), decode_smem_bytes(), stream, programmatic && cascade);
  return cascade ? cudaLaunchKernelEx(&lc.cfg, decode_kernel<4>, kmap, vmap, p)
                 : cudaLaunchKernelEx(&lc.cfg, decode_kernel<1>, kmap, vmap, p);
}

cudaError_t prepare_decode_kernels(int* blocks_per_sm_decode, int* blocks_per_sm_cascade) {
  cudaError_t e;
  e = cudaFuncSetAttribute(decode_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)decode_smem_bytes());
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(decode_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)decode_smem_bytes());
  if (e != cudaSuccess) return e;
  // the same (largest) shared-memory carveout as the append kernel, so that
  // decode CTAs can share an SM with an append CTA
  e = cudaFuncSetAttribute(decode_kernel<1>, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(decode_kernel<4>, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm_decode, decode_kernel<1>, kDecodeWarps * 32,
                                                    decode_smem_bytes());
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm_cascade, decode_kernel<4>, kDecodeWarps * 32,
                                                       decode_smem_bytes());
}

}  // namespace mcpu
