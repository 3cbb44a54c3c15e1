// Causal append-chunk attention on the 5th-generation tensor cores
// (tcgen05 + TMEM), for rows that append a tool-observation chunk (L > 1).
//
// One CTA per SM, persistent, 10 warps:
//   warps 0-7  softmax, two warpgroups over the same 128-row tile: thread t of
//              warpgroup h owns query row t & 127 (TMEM lane) and keys
//              64h..64h+63 of every 128-key block. Each warpgroup runs its own
//              online softmax over its half of the keys (running max, row
//              sum, lazy rescale of its own O accumulator when the max grows
//              by more than 2^8) and writes its 64 probabilities (bf16) to a
//              TMEM P buffer. The two halves meet once per tile, in the
//              epilogue: the partner threads swap (max, sum) through shared
//              memory, and each warpgroup combines O_0 and O_1 for 32 of the
//              64 output dims;
//   warp 8     TMA producer: item queue, the query tile (3-D box of
//              16 tokens x 8 heads x 64 dims) and a 4-stage ring of K/V
//              blocks (8 pages = 128 keys, 16 KiB each for K and V);
//   warp 9     MMA issuer: S_b = Q K_b^T (M 128, N 128, K 64; both operands
//              K-major from shared memory) into one of two TMEM S buffers,
//              then O_h += P_{b-1,h} V_{b-1,h} for h = 0, 1 (M 128, N 64,
//              K 64 each; P from TMEM, V MN-major from shared memory), the
//              two accumulation chains interleaved.
// A query tile is (128 / g) consecutive tokens x the g query heads of one kv
// head, so every row of the tile reads the same K/V stream. TMEM (512
// columns): S0, S1 (128 each), O_0, O_1, P0, P1 (64 each). P has buffers of
// its own, so an S buffer is free again as soon as the softmax has loaded it:
// S_{b+1} never waits for PV_{b-1}.
//
// Ordering (all mbarriers, all waits bounded):
//   kv_full/kv_empty   TMA ring; a stage is released by the commit after PV_b
//   s_full[2]          S_b complete (commit after the 4 QK^T MMAs)
//   s_free[2]          S_b loaded into registers (8 softmax warps arrive)
//   p_full[2]          P_b stored and O_h rescaled (8 softmax warps arrive)
//   o_ready[2]         PV_b complete, on barrier b & 1 (one phase per two
//                      blocks: a waiter is never two phases behind)
//   xchg[4][2]         (max, sum) swap of a warp pair (w, w + 4) in the
//                      epilogue, double-buffered by tile parity
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
constexpr int kTcSoftmaxWarps = 8;
constexpr int kTcProducerWarp = 8, kTcMmaWarp = 9;
constexpr int kTcThreads = 320;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS0 = 0, kColS1 = 128, kColO0 = 256, kColO1 = 320, kColP0 = 384, kColP1 = 448;
constexpr float kRescaleThreshold = 8.f;  // log2 units: P may reach 2^8 before O is rescaled

struct TcSmem {  // barriers and small state, after the tiles
  uint64_t q_full, q_empty, o_free;
  uint64_t o_ready[2];
  uint64_t kv_full[kTcStages], kv_empty[kTcStages];
  uint64_t s_full[2], s_free[2], p_full[2];
  uint64_t item_full[2], item_empty[2];
  uint64_t xchg[4][2];
  float2 xval[2][2][kTcRows];  // (max, sum) by [tile parity][warpgroup][row]
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
    mbar_init(bar(st.o_free), kTcSoftmaxWarps);
    for (int s = 0; s < kTcStages; ++s) {
      mbar_init(bar(st.kv_full[s]), 1);
      mbar_init(bar(st.kv_empty[s]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(st.s_full[i]), 1);
      mbar_init(bar(st.s_free[i]), kTcSoftmaxWarps);
      mbar_init(bar(st.o_ready[i]), 1);
      mbar_init(bar(st.p_full[i]), kTcSoftmaxWarps);
      mbar_init(bar(st.item_full[i]), 1);
      mbar_init(bar(st.item_empty[i]), kTcSoftmaxWarps + 1);
    }
    for (int w = 0; w < 4; ++w)
      for (int i = 0; i < 2; ++i) mbar_init(bar(st.xchg[w][i]), 2);
    st.abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == kTcMmaWarp) {
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

  if (warp == kTcProducerWarp) {
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
  } else if (warp == kTcMmaWarp) {
    // ----------------------------------------------------------- MMA issuer
    // Kept lean: the issue of consecutive tcgen05.mma is the critical path,
    // so descriptors are computed once per stage and stepped by constants.
    if (lane == 0) {
      constexpr uint32_t idS = idesc_bf16(kTcRows, kTcKeys, false, false);
      constexpr uint32_t idO = idesc_bf16(kTcRows, kHeadDim, false, true);
      // descriptors of stage 0; stage s starts s * kTcStageBytes further on
      // (the start-address field counts 16-byte units and cannot overflow:
      // shared memory ends below 256 KiB)
      const uint64_t qdesc = smem_desc_sw128(sQ, 16, 1024);
      const uint64_t kdesc0 = smem_desc_sw128(sKV, 16, 1024);
      const uint64_t vdesc0 = smem_desc_sw128(sKV + kTcKvBytes, 1024, 1024);
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
        // O += P_gblk V_gblk (b: block index within the item)
        auto issue_pv = [&](int b, uint32_t gblk, uint32_t it) -> bool {
          const uint32_t buf = gblk & 1;
          if (!wait_bar(bar(st.p_full[buf]), (gblk >> 1) & 1, abort_flag)) return false;
          if (b == 0 && i >= 1 && !wait_bar(bar(st.o_free), (i - 1) & 1, abort_flag)) return false;
          tc_fence_after();
          const int s = it % kTcStages;
          const uint32_t pcol = tmem + (buf ? kColP1 : kColP0);
          const uint64_t vd = vdesc0 + (uint64_t)(s * (kTcStageBytes / 16));
          // keys 0..63 into O_0, keys 64..127 into O_1, alternating
          constexpr uint64_t kStep = 16 * kRowBytes / 16;  // 16 keys of V, in 16-byte units
          tc_mma_ts(tmem + kColO0, pcol, vd, idO, b > 0 ? 1u : 0u);
          tc_mma_ts(tmem + kColO1, pcol + 32, vd + 4 * kStep, idO, b > 0 ? 1u : 0u);
#pragma unroll
          for (int kk = 1; kk < 4; ++kk) {
            tc_mma_ts(tmem + kColO0, pcol + kk * 8, vd + kk * kStep, idO, 1u);
            tc_mma_ts(tmem + kColO1, pcol + 32 + kk * 8, vd + (4 + kk) * kStep, idO, 1u);
          }
          tc_commit(bar(st.kv_empty[s]));
          tc_commit(bar(st.o_ready[buf]));
          return true;
        };
        for (int b = 0; b < nb; ++b, ++kv_it, ++blk) {
          const int s = kv_it % kTcStages;
          const uint32_t buf = blk & 1;
          if (!wait_bar(bar(st.kv_full[s]), (kv_it / kTcStages) & 1, abort_flag)) {
            ok = false;
            break;
          }
          // S buffer `buf` was last loaded by the softmax of block blk - 2
          if (blk >= 2 && !wait_bar(bar(st.s_free[buf]), ((blk - 2) >> 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t scol = tmem + (buf ? kColS1 : kColS0);
          const uint64_t kd = kdesc0 + (uint64_t)(s * (kTcStageBytes / 16));
          tc_mma_ss(scol, qdesc, kd, idS, 0u);
#pragma unroll
          for (int kk = 1; kk < kHeadDim / 16; ++kk)
            tc_mma_ss(scol, qdesc + (uint64_t)(kk * 2), kd + (uint64_t)(kk * 2), idS, 1u);
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
    const int row = threadIdx.x & (kTcRows - 1);  // TMEM lane
    const int half = threadIdx.x >> 7;            // keys 64*half .. +63 of a block
    const int wq = warp & 3;                      // TMEM lane quarter; pair (wq, wq + 4)
    const uint32_t lane_off = (uint32_t)(wq * 32) << 16;
    const uint32_t cO = half ? kColO1 : kColO0;   // this warpgroup's accumulator
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
      const int wp_min = a.pos_begin + min((wq * 32) / g, max(a.n_tok - 1, 0));
      const int wp_max = a.pos_begin + min((wq * 32 + 31) / g, max(a.n_tok - 1, 0));
      float m_ref = -INFINITY, l = 0.f;
      for (int b = 0; b < nb; ++b, ++blk) {
        const uint32_t buf = blk & 1;
        const uint32_t cS = (buf ? kColS1 : kColS0) + 64 * half;
        ok = __all_sync(0xffffffffu, wait_bar(bar(st.s_full[buf]), (blk >> 1) & 1, abort_flag));
        if (!ok) break;
        tc_fence_after();
        uint32_t sv[2][32];
        tmem_ld32(tmem + lane_off + cS, sv[0]);
        tmem_ld32(tmem + lane_off + cS + 32, sv[1]);
        tmem_ld_wait();
        // the scores are in registers: the S buffer may take block blk + 2
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(st.s_free[buf]));
        const int kbase = kb0 + b * kTcKeys + 64 * half;
        const bool need_mask = (kbase + 63 > wp_min) || (p.window > 0 && kbase < wp_max - p.window + 1);
        if (need_mask) {
#pragma unroll
          for (int c = 0; c < 2; ++c)
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              const int j = kbase + 32 * c + e;
              if (j > pos || j < lo) sv[c][e] = 0xff800000u;  // -inf
            }
        }
        // max of the raw scores of this half row (the scale is positive)
        float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int c = 0; c < 2; ++c)
#pragma unroll
          for (int e = 0; e < 32; e += 8)
#pragma unroll
            for (int k = 0; k < 4; ++k)
              mx4[k] = fmax3(mx4[k], __uint_as_float(sv[c][e + 2 * k]), __uint_as_float(sv[c][e + 2 * k + 1]));
        const float mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3])) * p.scale_log2;
        float alpha = 1.f;
        if (mx > m_ref + kRescaleThreshold) {  // also true for the first finite max
          alpha = ex2_approx(m_ref - mx);      // 0 when m_ref == -inf
          m_ref = mx;
        }
        const float neg_mu = m_ref == -INFINITY ? 0.f : -m_ref;
        // p = 2^(s * scale * log2e - m): the argument in packed pairs
        const uint64_t sl2x2 = pack_f32x2(p.scale_log2, p.scale_log2);
        const uint64_t nmux2 = pack_f32x2(neg_mu, neg_mu);
        uint64_t lsum[2] = {0, 0};  // four partial sums
        uint32_t pk[32];
#pragma unroll
        for (int c = 0; c < 2; ++c) {
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            const uint64_t x = fma2((uint64_t)sv[c][e] | ((uint64_t)sv[c][e + 1] << 32), sl2x2, nmux2);
            const float p0 = ex2_approx(lo_f32(x));
            const float p1 = ex2_approx(hi_f32(x));
            lsum[(e >> 1) & 1] = add2(lsum[(e >> 1) & 1], pack_f32x2(p0, p1));
            pk[c * 16 + e / 2] = pack_bf16x2(p0, p1);
          }
        }
        const uint64_t ls = add2(lsum[0], lsum[1]);
        l = l * alpha + (lo_f32(ls) + hi_f32(ls));
        // O_h may only be rescaled once PV_{blk-1} has completed
        if (b > 0 && __any_sync(0xffffffffu, alpha != 1.f)) {
          ok = __all_sync(0xffffffffu,
                          wait_bar(bar(st.o_ready[(blk - 1) & 1]), ((blk - 1) >> 1) & 1, abort_flag));
          if (!ok) break;
          tc_fence_after();
          uint32_t ov[2][32];
          tmem_ld32(tmem + lane_off + cO, ov[0]);
          tmem_ld32(tmem + lane_off + cO + 32, ov[1]);
          tmem_ld_wait();
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int e = 0; e < 32; ++e) ov[h][e] = __float_as_uint(__uint_as_float(ov[h][e]) * alpha);
          tmem_st32(tmem + lane_off + cO, ov[0]);
          tmem_st32(tmem + lane_off + cO + 32, ov[1]);
        }
        // P buffer `buf` was last read by PV_{blk-2}
        if (blk >= 2) {
          ok = __all_sync(0xffffffffu, wait_bar(bar(st.o_ready[buf]), ((blk - 2) >> 1) & 1, abort_flag));
          if (!ok) break;
          tc_fence_after();
        }
        tmem_st32(tmem + lane_off + (buf ? kColP1 : kColP0) + 32 * half, pk);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(st.p_full[buf]));
      }
      if (!ok) break;
      // epilogue: the last PV of the item, then combine the two halves
      if (nb > 0) {
        ok = __all_sync(0xffffffffu,
                        wait_bar(bar(st.o_ready[(blk - 1) & 1]), ((blk - 1) >> 1) & 1, abort_flag));
        if (!ok) break;
      }
      tc_fence_after();
      uint32_t o0[32], o1[32];  // dims 32*half..+31 of O_0 and O_1
      tmem_ld32(tmem + lane_off + kColO0 + 32 * half, o0);
      tmem_ld32(tmem + lane_off + kColO1 + 32 * half, o1);
      tmem_ld_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bar(st.o_free));
        mbar_arrive(bar(st.item_empty[slot]));
      }
      // swap (max, sum) with the partner thread of the other warpgroup
      const uint32_t par = i & 1;
      st.xval[par][half][row] = make_float2(m_ref, l);
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(st.xchg[wq][par]));
      ok = __all_sync(0xffffffffu, wait_bar(bar(st.xchg[wq][par]), (i >> 1) & 1, abort_flag));
      if (!ok) break;
      const float2 other = st.xval[par][half ^ 1][row];
      const float m0 = half ? other.x : m_ref, l0 = half ? other.y : l;
      const float m1 = half ? m_ref : other.x, l1 = half ? l : other.y;
      const float M = fmaxf(m0, m1);
      const float a0 = m0 == -INFINITY ? 0.f : ex2_approx(m0 - M);
      const float a1 = m1 == -INFINITY ? 0.f : ex2_approx(m1 - M);
      const float lt = l0 * a0 + l1 * a1;
      if (valid) {
        const float inv = lt > 0.f ? 1.f / lt : 0.f;
        const float w0 = a0 * inv, w1 = a1 * inv;
        const size_t orow = (size_t)(a.token_begin + tok) * Hq + kvh * g + head;
        uint4* dst = reinterpret_cast<uint4*>(p.out + orow * kHeadDim + 32 * half);
        auto o = [&](int e) { return __uint_as_float(o0[e]) * w0 + __uint_as_float(o1[e]) * w1; };
#pragma unroll
        for (int v = 0; v < 4; ++v) {
          const int e0 = v * 8;
          uint4 w;
          w.x = pack_bf16x2(o(e0 + 0), o(e0 + 1));
          w.y = pack_bf16x2(o(e0 + 2), o(e0 + 3));
          w.z = pack_bf16x2(o(e0 + 4), o(e0 + 5));
          w.w = pack_bf16x2(o(e0 + 6), o(e0 + 7));
          dst[v] = w;
        }
        if (half == 0) p.lse[orow] = lt > 0.f ? (M + __log2f(lt)) * 0.69314718055994531f : -INFINITY;
      }
    }
  }

  // every role ends here; a timed-out role has set the abort flag
  __syncwarp();
  if (threadIdx.x == 0 && *abort_flag) raise_status(p, kStatusTimeout);
  tc_fence_before();
  __syncthreads();
  if (warp == kTcMmaWarp) {
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
