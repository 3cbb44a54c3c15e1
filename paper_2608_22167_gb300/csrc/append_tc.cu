// Causal append-chunk attention on the 5th-generation tensor cores
// (tcgen05 + TMEM), for rows that append a tool-observation chunk (L > 1).
//
// One CTA per SM, persistent, 6 warps:
//   warps 0-3  softmax: thread t owns query row t of the 128-row tile (TMEM
//              lane t): reads S from TMEM, masks, keeps the running max and
//              row sum in registers, writes P (bf16) back over S, rescales O
//              in TMEM when the max grows by more than 2^8, and finally
//              normalises O and writes out / lse;
//   warp 4     TMA producer: item queue, the query tile (3-D box of
//              16 tokens x 8 heads x 64 dims) and a 4-stage ring of K/V
//              blocks (8 pages = 128 keys, 16 KiB each for K and V);
//   warp 5     MMA issuer: S_b = Q K_b^T (M 128, N 128, K 64; both operands
//              K-major from shared memory) into one of two TMEM S buffers,
//              then O += P_b V_b (M 128, N 64, K 128; P from TMEM, V MN-major
//              from shared memory) into a TMEM O accumulator.
// A query tile is (128 / g) consecutive tokens x the g query heads of one kv
// head, so every row of the tile reads the same K/V stream. TMEM: two S
// buffers of 128 columns and O of 64 columns (512 allocated).
//
// Ordering (all mbarriers, all waits bounded):
//   kv_full/kv_empty   TMA ring; a stage is released by the commit after PV_b
//   s_full[2]          S_b complete (commit after the 4 QK^T MMAs)
//   p_full[2]          P_b stored and O rescaled (4 softmax warps arrive)
//   o_ready[2]         PV_b complete, on barrier b & 1 (one phase per two blocks:
//                      a waiter is never two phases behind, even across the
//                      item boundary where PV_{b-1} is issued before S_{b+1})
//   q_full/q_empty     query tile loaded / last QK^T of the item done
//   o_free             epilogue has read O (next item may overwrite it)
//   item_full/empty[2] two-slot queue of work items from the producer
#include "tcgen05.cuh"

namespace mcpu {

constexpr int kTcRows = 128;         // query rows per tile (TMEM lanes)
constexpr int kTcKeys = 128;         // keys per block
constexpr int kTcStages = 4;
constexpr int kTcQBytes = kTcRows * kRowBytes;       // 16 KiB
constexpr int kTcKvBytes = kTcKeys * kRowBytes;      // 16 KiB each for K and V
constexpr int kTcStageBytes = 2 * kTcKvBytes;
constexpr int kTcThreads = 192;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS0 = 0, kColS1 = 128, kColO = 256;
constexpr float kRescaleThreshold = 8.f;  // log2 units: P may reach 2^8 before O is rescaled

struct TcSmem {  // barriers and small state, after the tiles
  uint64_t q_full, q_empty, o_free;
  uint64_t o_ready[2];
  uint64_t kv_full[kTcStages], kv_empty[kTcStages];
  uint64_t s_full[2], p_full[2];
  uint64_t item_full[2], item_empty[2];
  AppendItem items[2];
  int32_t item_idx[2];
  uint32_t tmem_base;
  int32_t abort_flag;
};

size_t append_tc_smem_bytes() { return 1024 + kTcQBytes + (size_t)kTcStages * kTcStageBytes + sizeof(TcSmem); }

namespace {

// Bounded wait that also gives up when another role has aborted.
__device__ __forceinline__ bool wait_bar(uint32_t bar, uint32_t parity, volatile int32_t* abort_flag) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (*abort_flag) return false;
    if (global_timer_ns() - t0 > kWaitTimeoutNs) {
      *abort_flag = 1;
      return false;
    }
  }
  return true;
}

}  // namespace

__global__ void __launch_bounds__(kTcThreads, 1)
    append_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                     const __grid_constant__ CUtensorMap qmap, const AttnParams p) {
  extern __shared__ uint8_t smem_raw[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t raw = smem_addr(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t sQ = base;
  const uint32_t sKV = base + kTcQBytes;
  TcSmem& st = *reinterpret_cast<TcSmem*>(smem_raw + (base - raw) + kTcQBytes + kTcStages * kTcStageBytes);
  volatile int32_t* abort_flag = &st.abort_flag;
  auto bar = [&](uint64_t& b) { return smem_addr(&b); };

  if (threadIdx.x == 0) {
    mbar_init(bar(st.q_full), 1);
    mbar_init(bar(st.q_empty), 1);
    mbar_init(bar(st.o_free), 4);
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(bar(st.kv_full[s]), 1);
      mbar_init(bar(st.kv_empty[s]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(st.s_full[i]), 1);
      mbar_init(bar(st.o_ready[i]), 1);
      mbar_init(bar(st.p_full[i]), 4);
      mbar_init(bar(st.item_full[i]), 1);
      mbar_init(bar(st.item_empty[i]), 5);
    }
    st.abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 5) {
    tmem_alloc(smem_addr(&st.tmem_base), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = st.tmem_base;

  PlanHeader* hdr = header(p);
  const int Hkv = p.num_kv_heads, Hq = p.num_q_heads, g = p.group;
  const int n_items = hdr->n_append * Hkv;
  const AppendItem* items = reinterpret_cast<const AppendItem*>(p.ws + p.lay.append_items);

  if (warp == 4) {
    // ------------------------------------------------------------ producer
    // The whole warp runs this loop: lane i keeps the page id of page
    // (chunk + i) for the current and the next 32-page chunk, so the block
    // table is read ahead with coalesced loads; lane 0 issues the copies.
    if (lane == 0) {
      prefetch_tensormap(&kmap);
      prefetch_tensormap(&vmap);
      prefetch_tensormap(&qmap);
    }
    const uint64_t pol = policy_evict_last();
    uint32_t kv_it = 0;
    for (int i = 0;; ++i) {
      const int slot = i & 1;
      if (i >= 2 && !__all_sync(0xffffffffu, wait_bar(bar(st.item_empty[slot]), ((i >> 1) - 1) & 1, abort_flag)))
        break;
      int idx = 0;
      if (lane == 0) idx = atomicAdd(&hdr->append_ticket, 1);
      idx = __shfl_sync(0xffffffffu, idx, 0);
      AppendItem a;
      if (idx < n_items) a = items[idx / Hkv];
      if (lane == 0) {
        st.item_idx[slot] = idx;
        st.items[slot] = a;
        mbar_arrive(bar(st.item_full[slot]));
      }
      if (idx >= n_items) break;
      const int kvh = idx % Hkv;
      const int* bt_row = p.block_table + (size_t)a.row * p.max_pages;
      const int pg0 = a.key_begin / kPage;
      const int kb0 = pg0 * kPage;
      const int nb = (a.key_end - kb0 + kTcKeys - 1) / kTcKeys;
      const int page_end = (a.key_end + kPage - 1) / kPage;
      auto load_chunk = [&](int c) -> int {  // page id of page pg0 + 32c + lane, or -1
        const int lp = pg0 + 32 * c + lane;
        int v = -1;
        if (lp < page_end) {
          v = __ldg(bt_row + lp);
          if (v < 0 || v >= p.num_pages) {
            raise_status(p, kStatusBadPage);
            v = -1;
          }
        }
        return v;
      };
      int pid_cur = load_chunk(0), pid_next = load_chunk(1);
      if (i >= 1 && !__all_sync(0xffffffffu, wait_bar(bar(st.q_empty), (i - 1) & 1, abort_flag))) break;
      if (lane == 0) {
        mbar_arrive_expect_tx(bar(st.q_full), kTcQBytes);
        tma_load_3d(sQ, &qmap, 0, kvh * g, a.token_begin, bar(st.q_full));
      }
      bool ok = true;
      constexpr int kPagesPerBlock = kTcKeys / kPage;  // 8: four blocks per 32-page chunk
      for (int b = 0; b < nb; ++b, ++kv_it) {
        if (b > 0 && (b * kPagesPerBlock) % 32 == 0) {
          pid_cur = pid_next;
          pid_next = load_chunk(b * kPagesPerBlock / 32 + 1);
        }
        const int s = kv_it % kTcStages;
        if (kv_it >= kTcStages &&
            !__all_sync(0xffffffffu, wait_bar(bar(st.kv_empty[s]), ((kv_it / kTcStages) - 1) & 1, abort_flag))) {
          ok = false;
          break;
        }
        const uint32_t dk = sKV + s * kTcStageBytes, dv = dk + kTcKvBytes;
        const int lane0 = (b * kPagesPerBlock) % 32;
        int y[kPagesPerBlock];
#pragma unroll
        for (int j = 0; j < kPagesPerBlock; ++j) {
          const int pid = __shfl_sync(0xffffffffu, pid_cur, lane0 + j);
          y[j] = pid < 0 ? p.oob_row : (pid * Hkv + kvh) * kPage;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(bar(st.kv_full[s]), kTcStageBytes);
#pragma unroll
          for (int j = 0; j < kPagesPerBlock; ++j) {
            tma_load_2d(dk + j * kTileBytes, &kmap, 0, y[j], bar(st.kv_full[s]), pol);
            tma_load_2d(dv + j * kTileBytes, &vmap, 0, y[j], bar(st.kv_full[s]), pol);
          }
        }
      }
      if (!ok) break;
    }
  } else if (warp == 5) {
    // ----------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idS = idesc_bf16(kTcRows, kTcKeys, false, false);
      constexpr uint32_t idO = idesc_bf16(kTcRows, kHeadDim, false, true);
      uint32_t kv_it = 0, blk = 0;
      bool ok = true;
      for (int i = 0; ok; ++i) {
        const int slot = i & 1;
        if (!wait_bar(bar(st.item_full[slot]), (i >> 1) & 1, abort_flag)) break;
        const int idx = st.item_idx[slot];
        const AppendItem a = st.items[slot];
        if (idx >= n_items) break;
        const int kb0 = (a.key_begin / kPage) * kPage;
        const int nb = (a.key_end - kb0 + kTcKeys - 1) / kTcKeys;
        if (!wait_bar(bar(st.q_full), i & 1, abort_flag)) break;
        tc_fence_after();
        const uint64_t qdesc = smem_desc_sw128(sQ, 16, 1024);
        auto issue_pv = [&](int b, uint32_t gblk, uint32_t it) -> bool {
          const uint32_t buf = gblk & 1;
          if (!wait_bar(bar(st.p_full[buf]), (gblk >> 1) & 1, abort_flag)) return false;
          if (b == 0 && i >= 1 && !wait_bar(bar(st.o_free), (i - 1) & 1, abort_flag)) return false;
          tc_fence_after();
          const int s = it % kTcStages;
          const uint32_t sv = sKV + s * kTcStageBytes + kTcKvBytes;
#pragma unroll
          for (int kk = 0; kk < kTcKeys / 16; ++kk) {
            const uint64_t vdesc = smem_desc_sw128(sv + kk * 16 * kRowBytes, 1024, 1024);
            tc_mma_ts(tmem + kColO, tmem + (buf ? kColS1 : kColS0) + kk * 8, vdesc, idO, (b > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(bar(st.kv_empty[s]));
          tc_commit(bar(st.o_ready[gblk & 1]));
          return true;
        };
        for (int b = 0; b < nb; ++b, ++kv_it, ++blk) {
          const int s = kv_it % kTcStages;
          const uint32_t buf = blk & 1;
          if (!wait_bar(bar(st.kv_full[s]), (kv_it / kTcStages) & 1, abort_flag)) {
            ok = false;
            break;
          }
          // S buffer `buf` was last read by PV_{blk-2}: wait for it
          if (blk >= 2 && !wait_bar(bar(st.o_ready[blk & 1]), ((blk - 2) >> 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sk = sKV + s * kTcStageBytes;
#pragma unroll
          for (int kk = 0; kk < kHeadDim / 16; ++kk) {
            const uint64_t kdesc = smem_desc_sw128(sk + kk * 32, 16, 1024);
            tc_mma_ss(tmem + (buf ? kColS1 : kColS0), qdesc + (uint64_t)(kk * 2), kdesc, idS, kk > 0 ? 1u : 0u);
          }
          tc_commit(bar(st.s_full[buf]));
          if (b == nb - 1) tc_commit(bar(st.q_empty));
          if (b >= 1 && !issue_pv(b - 1, blk - 1, kv_it - 1)) {
            ok = false;
            break;
          }
        }
        if (!ok) break;
        if (nb > 0 && !issue_pv(nb - 1, blk - 1, kv_it - 1)) break;
        mbar_arrive(bar(st.item_empty[slot]));
      }
    }
  } else {
    // ------------------------------------------------------------- softmax
    const int row = threadIdx.x;  // 0..127 == TMEM lane
    const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
    uint32_t blk = 0;
    bool ok = true;
    for (int i = 0; ok; ++i) {
      const int slot = i & 1;
      ok = __all_sync(0xffffffffu, wait_bar(bar(st.item_full[slot]), (i >> 1) & 1, abort_flag));
      if (!ok) break;
      const int idx = st.item_idx[slot];
      const AppendItem a = st.items[slot];
      if (idx >= n_items) break;
      const int kvh = idx % Hkv;
      const int tok = row / g, head = row % g;
      const bool valid = tok < a.n_tok;
      const int pos = a.pos_begin + (valid ? tok : 0);
      const int lo = p.window > 0 ? pos - p.window + 1 : 0;
      const int kb0 = (a.key_begin / kPage) * kPage;
      const int nb = (a.key_end - kb0 + kTcKeys - 1) / kTcKeys;
      // warp-uniform position range of this warp's rows, for mask skipping
      const int wtok_lo = (warp * 32) / g;
      const int wp_min = a.pos_begin + min(wtok_lo, max(a.n_tok - 1, 0));
      const int wp_max = a.pos_begin + min((warp * 32 + 31) / g, max(a.n_tok - 1, 0));
      float m_ref = -INFINITY, l = 0.f;
      for (int b = 0; b < nb; ++b, ++blk) {
        const uint32_t buf = blk & 1;
        const uint32_t cS = buf ? kColS1 : kColS0;
        ok = __all_sync(0xffffffffu, wait_bar(bar(st.s_full[buf]), (blk >> 1) & 1, abort_flag));
        if (!ok) break;
        tc_fence_after();
        uint32_t sv[4][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32(tmem + lane_off + cS + 32 * c, sv[c]);
        tmem_ld_wait();
        const int kbase = kb0 + b * kTcKeys;
        const bool need_mask = (kbase + kTcKeys - 1 > wp_min) || (p.window > 0 && kbase < wp_max - p.window + 1);
        if (need_mask) {
#pragma unroll
          for (int c = 0; c < 4; ++c)
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              const int j = kbase + 32 * c + e;
              if (j > pos || j < lo) sv[c][e] = 0xff800000u;  // -inf
            }
        }
        // row max of the raw scores (the scale is positive), two chains
        float mxa = -INFINITY, mxb = -INFINITY;
#pragma unroll
        for (int c = 0; c < 4; ++c)
#pragma unroll
          for (int e = 0; e < 32; e += 4) {
            mxa = fmax3(mxa, __uint_as_float(sv[c][e]), __uint_as_float(sv[c][e + 1]));
            mxb = fmax3(mxb, __uint_as_float(sv[c][e + 2]), __uint_as_float(sv[c][e + 3]));
          }
        const float mx = fmaxf(mxa, mxb) * p.scale_log2;
        float alpha = 1.f;
        if (mx > m_ref + kRescaleThreshold) {  // also true for the first finite max
          alpha = ex2_approx(m_ref - mx);      // 0 when m_ref == -inf
          m_ref = mx;
        }
        const float neg_mu = m_ref == -INFINITY ? 0.f : -m_ref;
        // p = 2^(s * scale * log2e - m): the argument in packed pairs
        const uint64_t sl2x2 = pack_f32x2(p.scale_log2, p.scale_log2);
        const uint64_t nmux2 = pack_f32x2(neg_mu, neg_mu);
        uint64_t lsum = 0;  // two partial row sums
        uint32_t pk[2][32];
#pragma unroll
        for (int c = 0; c < 4; ++c) {
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const uint64_t x = fma2((uint64_t)sv[c][e] | ((uint64_t)sv[c][e + 1] << 32), sl2x2, nmux2);
            const float p0 = ex2_approx(lo_f32(x));
            const float p1 = ex2_approx(hi_f32(x));
            lsum = add2(lsum, pack_f32x2(p0, p1));
            pk[c >> 1][(c & 1) * 16 + e / 2] = pack_bf16x2(p0, p1);
          }
        }
        const float la = lo_f32(lsum), lb = hi_f32(lsum);
        l = l * alpha + (la + lb);
        // O may only be rescaled once PV_{blk-1} has completed. Without a
        // rescale P_blk is published right away: PV_blk queues behind
        // PV_{blk-1} on the tensor pipe.
        if (b > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
          ok = __all_sync(0xffffffffu,
                          wait_bar(bar(st.o_ready[(blk - 1) & 1]), ((blk - 1) >> 1) & 1, abort_flag));
          if (!ok) break;
          tc_fence_after();
          uint32_t ov[2][32];
          tmem_ld32(tmem + lane_off + kColO, ov[0]);
          tmem_ld32(tmem + lane_off + kColO + 32, ov[1]);
          tmem_ld_wait();
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[h][e] = __float_as_uint(__uint_as_float(ov[h][e]) * alpha);
          tmem_st32(tmem + lane_off + kColO, ov[0]);
          tmem_st32(tmem + lane_off + kColO + 32, ov[1]);
        }
        tmem_st32(tmem + lane_off + cS, pk[0]);
        tmem_st32(tmem + lane_off + cS + 32, pk[1]);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(st.p_full[buf]));
      }
      if (!ok) break;
      // epilogue: the last PV of the item
      if (nb > 0) {
        ok = __all_sync(0xffffffffu,
                        wait_bar(bar(st.o_ready[(blk - 1) & 1]), ((blk - 1) >> 1) & 1, abort_flag));
        if (!ok) break;
      }
      tc_fence_after();
      uint32_t ov[2][32];
      tmem_ld32(tmem + lane_off + kColO, ov[0]);
      tmem_ld32(tmem + lane_off + kColO + 32, ov[1]);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bar(st.o_free));
        mbar_arrive(bar(st.item_empty[slot]));
      }
      if (valid) {
        const float inv = l > 0.f ? 1.f / l : 0.f;
        const size_t orow = (size_t)(a.token_begin + tok) * Hq + kvh * g + head;
        uint4* dst = reinterpret_cast<uint4*>(p.out + orow * kHeadDim);
#pragma unroll
        for (int v = 0; v < 8; ++v) {
          const int h = v >> 2, e0 = (v & 3) * 8;
          uint4 w;
          w.x = pack_bf16x2(__uint_as_float(ov[h][e0 + 0]) * inv, __uint_as_float(ov[h][e0 + 1]) * inv);
          w.y = pack_bf16x2(__uint_as_float(ov[h][e0 + 2]) * inv, __uint_as_float(ov[h][e0 + 3]) * inv);
          w.z = pack_bf16x2(__uint_as_float(ov[h][e0 + 4]) * inv, __uint_as_float(ov[h][e0 + 5]) * inv);
          w.w = pack_bf16x2(__uint_as_float(ov[h][e0 + 6]) * inv, __uint_as_float(ov[h][e0 + 7]) * inv);
          dst[v] = w;
        }
        p.lse[orow] = l > 0.f ? (m_ref + __log2f(l)) * 0.69314718055994531f : -INFINITY;
      }
    }
  }

  // every role ends here; a timed-out role has set the abort flag
  __syncwarp();
  if (threadIdx.x == 0 && *abort_flag) raise_status(p, kStatusTimeout);
  tc_fence_before();
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

cudaError_t launch_append_tc(const CUtensorMap& kmap, const CUtensorMap& vmap, const CUtensorMap& qmap,
                             const AttnParams& p, int grid, cudaStream_t stream) {
  append_tc_kernel<<<grid, kTcThreads, append_tc_smem_bytes(), stream>>>(kmap, vmap, qmap, p);
  return cudaGetLastError();
}

cudaError_t prepare_append_tc_kernel(int* blocks_per_sm) {
  cudaError_t e = cudaFuncSetAttribute(append_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)append_tc_smem_bytes());
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(append_tc_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                           cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(blocks_per_sm, append_tc_kernel, kTcThreads,
                                                       append_tc_smem_bytes());
}

}  // namespace mcpu
