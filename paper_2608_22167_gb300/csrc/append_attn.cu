// Causal append-chunk attention (rows with L > 1: a tool observation being
// appended, paper §3.2), flash-attention style on mma.sync tensor cores.
//
// A CTA tile is 64 query rows = (64 / g) consecutive tokens x the g query
// heads of one kv head, so all rows share the K/V stream. Four warps own 16
// rows each. K/V arrive in blocks of 64 keys (4 pages, 8 TMA loads of 2 KiB,
// 128-byte swizzle) through a 3-stage ring with full/empty mbarriers.
// Per block and warp: S = Q K^T (32 mma m16n8k16), causal + window mask on
// the blocks that straddle a boundary, online softmax in fp32 (base 2), then
// O += P V (32 mma) with P taken straight from the S accumulators.
// Tiles are handed out by an atomic ticket so long rows do not serialise.
#include "common.cuh"

namespace mcpu {

constexpr int kAppWarps = 4;
constexpr int kAppStages = 3;
constexpr int kKeyBlock = 64;                               // keys per stage
constexpr int kAppStageBytes = 2 * kKeyBlock * kRowBytes;  // K + V: 16 KiB

size_t append_smem_bytes() {
  return 1024 + (size_t)kAppStages * kAppStageBytes + kAppStages * 16 + 16;
}

__global__ void __launch_bounds__(kAppWarps * 32)
    append_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                  const AttnParams p) {
  if (header(p)->n_append == 0) return;  // no append rows this call
  extern __shared__ uint8_t smem_raw[];
  __shared__ int s_item;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t full = base + kAppStages * kAppStageBytes;  // kAppStages barriers
  const uint32_t empty = full + kAppStages * 8;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kAppStages; ++s) {
      mbar_init(full + 8 * s, 1);
      mbar_init(empty + 8 * s, kAppWarps);
    }
    fence_barrier_init();
    prefetch_tensormap(&kmap);
    prefetch_tensormap(&vmap);
  }
  __syncthreads();

  PlanHeader* hdr = header(p);
  const int Hkv = p.num_kv_heads, Hq = p.num_q_heads, g = p.group;
  const int n_items = hdr->n_append * Hkv;
  const AppendItem* items = reinterpret_cast<const AppendItem*>(p.ws + p.lay.append_items);
  const uint64_t pol = policy_evict_first();
  const int mi = lane >> 3, ri = lane & 7;
  uint32_t seq = 0;  // key blocks consumed by this CTA (ring position/phase)
  bool dead = false;

  while (true) {
    if (threadIdx.x == 0) s_item = atomicAdd(&hdr->append_ticket, 1);
    __syncthreads();
    const int it = s_item;
    __syncthreads();
    if (it >= n_items || dead) break;
    const int rec = it / Hkv, kvh = it % Hkv;
    const AppendItem a = items[rec];
    const int* bt_row = p.block_table + (size_t)a.row * p.max_pages;

    // this warp's two fragment rows: r0 = 16*warp + lane/4, r1 = r0 + 8
    const int r0 = warp * 16 + (lane >> 2), r1 = r0 + 8;
    const int tk0 = r0 / g, tk1 = r1 / g;
    const bool ok0 = tk0 < a.n_tok, ok1 = tk1 < a.n_tok;
    const int pos0 = a.pos_begin + (ok0 ? tk0 : 0), pos1 = a.pos_begin + (ok1 ? tk1 : 0);
    const int lo0 = p.window > 0 ? pos0 - p.window + 1 : 0, lo1 = p.window > 0 ? pos1 - p.window + 1 : 0;

    // Q as the A operand (rows x head dim), straight from global memory
    uint32_t qa[4][4];
    {
      const uint32_t* q0p = reinterpret_cast<const uint32_t*>(
          p.q + ((size_t)(a.token_begin + tk0) * Hq + kvh * g + r0 % g) * kHeadDim);
      const uint32_t* q1p = reinterpret_cast<const uint32_t*>(
          p.q + ((size_t)(a.token_begin + tk1) * Hq + kvh * g + r1 % g) * kHeadDim);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        qa[kk][0] = ok0 ? __ldg(q0p + kk * 8 + (lane & 3)) : 0u;
        qa[kk][1] = ok1 ? __ldg(q1p + kk * 8 + (lane & 3)) : 0u;
        qa[kk][2] = ok0 ? __ldg(q0p + kk * 8 + 4 + (lane & 3)) : 0u;
        qa[kk][3] = ok1 ? __ldg(q1p + kk * 8 + 4 + (lane & 3)) : 0u;
      }
    }
    // warp-uniform bounds of its rows' visible keys, for mask skipping
    const int wtok_lo = (warp * 16) / g;
    const int wtok_hi = min((warp * 16 + 15) / g, a.n_tok - 1);
    const int wp_min = a.pos_begin + wtok_lo, wp_max = a.pos_begin + max(wtok_hi, 0);

    const int kb0 = (a.key_begin / kPage) * kPage;
    const int n_blocks = (a.key_end - kb0 + kKeyBlock - 1) / kKeyBlock;
    const int page_end = (a.key_end + kPage - 1) / kPage;

    auto issue = [&](int b) {  // thread 0 only
      const uint32_t s = (seq + b) % kAppStages;
      const uint32_t ph = ((seq + b) / kAppStages) & 1u;
      if (seq + b >= kAppStages) {
        if (!mbar_wait(empty + 8 * s, ph ^ 1u)) {
          raise_status(p, kStatusTimeout);
          dead = true;
          return;
        }
      }
      mbar_arrive_expect_tx(full + 8 * s, kAppStageBytes);
      const uint32_t dst = base + s * kAppStageBytes;
#pragma unroll
      for (int i = 0; i < kKeyBlock / kPage; ++i) {
        const int lp = kb0 / kPage + b * (kKeyBlock / kPage) + i;
        int y = p.oob_row;
        if (lp < page_end) {
          const int pid = __ldg(bt_row + lp);
          if (pid < 0 || pid >= p.num_pages)
            raise_status(p, kStatusBadPage);
          else
            y = (pid * Hkv + kvh) * kPage;
        }
        tma_load_2d(dst + i * kTileBytes, &kmap, 0, y, full + 8 * s, pol);
        tma_load_2d(dst + kKeyBlock * kRowBytes + i * kTileBytes, &vmap, 0, y, full + 8 * s, pol);
      }
    };
    if (threadIdx.x == 0)
      for (int b = 0; b < n_blocks && b < kAppStages - 1; ++b) issue(b);

    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    float o[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;

    bool timed_out = false;
    for (int b = 0; b < n_blocks; ++b) {
      if (threadIdx.x == 0 && b + kAppStages - 1 < n_blocks && !dead) issue(b + kAppStages - 1);
      const uint32_t s = (seq + b) % kAppStages;
      const uint32_t ph = ((seq + b) / kAppStages) & 1u;
      if (!__any_sync(0xffffffffu, mbar_wait(full + 8 * s, ph))) {
        timed_out = true;
        break;
      }
      const uint32_t kt = base + s * kAppStageBytes, vt = kt + kKeyBlock * kRowBytes;
      const int kbase = kb0 + b * kKeyBlock;

      float sc[8][4];
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) sc[nt][0] = sc[nt][1] = sc[nt][2] = sc[nt][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
        for (int np = 0; np < 4; ++np) {
          uint32_t b0, b1, b2, b3;
          ldmatrix_x4(kt + swz128(np * 16 + ri + (mi >> 1) * 8, 2 * kk + (mi & 1)), b0, b1, b2, b3);
          mma_bf16_16816(sc[2 * np], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b0, b1);
          mma_bf16_16816(sc[2 * np + 1], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b2, b3);
        }
      }
      // mask: key j visible to a row at position pos iff lo <= j <= pos
      const bool need_mask = (kbase + kKeyBlock - 1 > wp_min) || (p.window > 0 && kbase < wp_max - p.window + 1);
      float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const int j = kbase + nt * 8 + 2 * (lane & 3) + e;
          float x0 = sc[nt][e] * p.scale_log2, x1 = sc[nt][e + 2] * p.scale_log2;
          if (need_mask) {
            if (j > pos0 || j < lo0) x0 = -INFINITY;
            if (j > pos1 || j < lo1) x1 = -INFINITY;
          }
          sc[nt][e] = x0;
          sc[nt][e + 2] = x1;
          mx0 = fmaxf(mx0, x0);
          mx1 = fmaxf(mx1, x1);
        }
      }
#pragma unroll
      for (int off = 1; off < 4; off <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
      }
      const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
      const float mu0 = mn0 == -INFINITY ? 0.f : mn0, mu1 = mn1 == -INFINITY ? 0.f : mn1;
      const float al0 = fast_exp2(m0 - mu0), al1 = fast_exp2(m1 - mu1);
      m0 = mn0;
      m1 = mn1;
      float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
      for (int nt = 0; nt < 8; ++nt) {
        sc[nt][0] = fast_exp2(sc[nt][0] - mu0);
        sc[nt][1] = fast_exp2(sc[nt][1] - mu0);
        sc[nt][2] = fast_exp2(sc[nt][2] - mu1);
        sc[nt][3] = fast_exp2(sc[nt][3] - mu1);
        rs0 += sc[nt][0] + sc[nt][1];
        rs1 += sc[nt][2] + sc[nt][3];
        o[nt][0] *= al0;
        o[nt][1] *= al0;
        o[nt][2] *= al1;
        o[nt][3] *= al1;
      }
      l0 = l0 * al0 + rs0;
      l1 = l1 * al1 + rs1;

      // V rows of slots outside [key_begin, key_end) (the partial first page
      // of a window, the partial last page) were perhaps never written and
      // may hold NaN, which a zero weight does not cancel: they are zeroed in
      // the operand. Per key step this lane's b0/b2 hold keys 2c, 2c + 1 and
      // b1/b3 keys 2c + 8, 2c + 9 (c = lane & 3), the lower key in the low half.
      const bool v_edge = kbase < a.key_begin || kbase + kKeyBlock > a.key_end;
      // O += P V, P from the S accumulators (key step ks covers keys 16ks..16ks+15)
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        const uint32_t pa0 = pack_bf16x2(sc[2 * ks][0], sc[2 * ks][1]);
        const uint32_t pa1 = pack_bf16x2(sc[2 * ks][2], sc[2 * ks][3]);
        const uint32_t pa2 = pack_bf16x2(sc[2 * ks + 1][0], sc[2 * ks + 1][1]);
        const uint32_t pa3 = pack_bf16x2(sc[2 * ks + 1][2], sc[2 * ks + 1][3]);
        uint32_t vm_lo = 0xffffffffu, vm_hi = 0xffffffffu;
        if (v_edge) {
          const int jv = kbase + ks * 16 + 2 * (lane & 3);
          auto seen = [&](int j) { return j >= a.key_begin && j < a.key_end; };
          vm_lo = (seen(jv) ? 0x0000ffffu : 0u) | (seen(jv + 1) ? 0xffff0000u : 0u);
          vm_hi = (seen(jv + 8) ? 0x0000ffffu : 0u) | (seen(jv + 9) ? 0xffff0000u : 0u);
        }
#pragma unroll
        for (int dp = 0; dp < 4; ++dp) {
          uint32_t b0, b1, b2, b3;
          ldmatrix_x4_trans(vt + swz128(ks * 16 + ri + (mi & 1) * 8, 2 * dp + (mi >> 1)), b0, b1, b2, b3);
          b0 &= vm_lo;
          b2 &= vm_lo;
          b1 &= vm_hi;
          b3 &= vm_hi;
          mma_bf16_16816(o[2 * dp], pa0, pa1, pa2, pa3, b0, b1);
          mma_bf16_16816(o[2 * dp + 1], pa0, pa1, pa2, pa3, b2, b3);
        }
      }
      fence_proxy_async();
      __syncwarp();
      if (lane == 0) mbar_arrive(empty + 8 * s);
    }
    if (__syncthreads_or(timed_out ? 1 : 0)) {
      raise_status(p, kStatusTimeout);
      return;  // ring phases are lost: the whole CTA stops
    }
    seq += n_blocks;

    // epilogue: normalise and write bf16 rows + lse
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, off);
      l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }
    float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
    float b0 = l0 > 0.f ? m0 + __log2f(l0) : -INFINITY, b1 = l1 > 0.f ? m1 + __log2f(l1) : -INFINITY;
    if (p.sinks != nullptr) {  // the sink joins the normaliser
      inv0 = finish_with_sink(m0, l0, sink_log2(p, kvh * g + r0 % g), &b0);
      inv1 = finish_with_sink(m1, l1, sink_log2(p, kvh * g + r1 % g), &b1);
    }
    const size_t orow0 = ((size_t)(a.token_begin + tk0) * Hq + kvh * g + r0 % g);
    const size_t orow1 = ((size_t)(a.token_begin + tk1) * Hq + kvh * g + r1 % g);
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      const int d = nt * 8 + 2 * (lane & 3);
      if (ok0)
        *reinterpret_cast<uint32_t*>(p.out + orow0 * kHeadDim + d) = pack_bf16x2(o[nt][0] * inv0, o[nt][1] * inv0);
      if (ok1)
        *reinterpret_cast<uint32_t*>(p.out + orow1 * kHeadDim + d) = pack_bf16x2(o[nt][2] * inv1, o[nt][3] * inv1);
    }
    if ((lane & 3) == 0) {
      if (ok0) p.lse[orow0] = b0 * 0.69314718055994531f;
      if (ok1) p.lse[orow1] = b1 * 0.69314718055994531f;
    }
  }
}

cudaError_t launch_append(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttnParams& p, int grid,
                          cudaStream_t stream) {
  append_kernel<<<grid, kAppWarps * 32, append_smem_bytes(), stream>>>(kmap, vmap, p);
  return cudaGetLastError();
}

cudaError_t prepare_append_kernel(int* blocks_per_sm) {
  cudaError_t e = cudaFuncSetAttribute(append_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)append_smem_bytes());
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(append_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, append_kernel, kAppWarps * 32,
                                                       append_smem_bytes());
}

}  // namespace mcpu
